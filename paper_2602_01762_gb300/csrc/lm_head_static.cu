// LM-head selection with no device allocation: the final RMSNorm, the shared
// LM-head projection and the top-k of a batch of hidden rows, run by the same
// GEMV + top-k kernel as the last stage of a draft step, with that kernel's
// scratch held in a static device array compiled into this library.
//
// Some callers cannot call cudaMalloc: an inference server whose caching
// allocator has already reserved the device memory it may use, a plugin whose
// host framework forbids allocation outside its own pool, or a process that
// fixes its whole device-memory budget at start-up.  They cannot create a
// prism_ctx (which owns a workspace), so this entry point takes only inputs
// and outputs and keeps its scratch here.
#include <cstdio>
#include <mutex>
#include <string>

#include "../../include/prism.h"
#include "common.cuh"

using namespace prism;

namespace {

constexpr int kStaticMaxRows = 64;    // hidden rows per call
constexpr int kStaticMaxGrid = 256;   // CTAs of the LM-head launch
constexpr int kMaxDevices = 64;
constexpr size_t kHeadBytes = 256;    // error word [0, 32), last-CTA ticket at 64
constexpr size_t kPartBytes = (size_t)kStaticMaxRows * kStaticMaxGrid * kTopK * 4;

// [head | partial top-8 values | partial top-8 ids], 1 MiB + 256 B.  Every
// process that loads the library holds it on every device it uses, until exit.
static __device__ __align__(256) unsigned char g_lm_scratch[kHeadBytes + 2 * kPartBytes];

struct DeviceState {
    bool ready = false;
    unsigned char *scratch = nullptr;   // device address of g_lm_scratch
    int sms = 0;
};

std::mutex g_setup_mutex;
DeviceState g_dev[kMaxDevices];

// Once per device, with that device current: resolve the array's device
// address (the host-side symbol is only a stand-in) and set the kernels'
// shared-memory attributes.
prism_status setup_device(int dev, DeviceState &out) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    DeviceState &st = g_dev[dev];
    if (!st.ready) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_lm_scratch);
        if (e != cudaSuccess) {
            set_global_error((std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e)).c_str());
            return PRISM_ERR_CUDA;
        }
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess) e = prepare_gemv_kernels();
        if (e != cudaSuccess) {
            set_global_error((std::string("device setup: ") + cudaGetErrorString(e)).c_str());
            return PRISM_ERR_CUDA;
        }
        st.scratch = (unsigned char *)p;
        st.sms = sms;
        st.ready = true;
    }
    out = st;
    return PRISM_OK;
}

prism_status reject(prism_status s, const std::string &msg) {
    set_global_error(msg.c_str());
    return s;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

// True when p is memory the current device dev can address as its own:
// device memory of dev, or managed memory.  Host pointers and other devices'
// memory are refused before any launch.
bool on_device(const void *p, int dev) {
    if (!p) return true;
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (at.type == cudaMemoryTypeManaged) return true;
    return at.type == cudaMemoryTypeDevice && at.device == dev;
}

}  // namespace

extern "C" prism_status prism_lm_head_topk_static(int32_t dtype, int32_t hidden, int32_t vocab,
                                                  int32_t batch, int32_t topk, float rms_eps,
                                                  const float *h, const void *g_final,
                                                  const void *lm_head, int32_t *draft,
                                                  int32_t *topk_ids, float *topk_logits,
                                                  float *logits, int32_t *dev_flags, void *stream) {
    if (dtype != PRISM_F32 && dtype != PRISM_BF16) return reject(PRISM_ERR_INVALID_ARG, "dtype must be PRISM_F32 or PRISM_BF16");
    if (!h || !lm_head || !draft) return reject(PRISM_ERR_INVALID_ARG, "h, lm_head and draft are required");
    if (!aligned16(h) || !aligned16(lm_head) || (g_final && !aligned16(g_final)))
        return reject(PRISM_ERR_INVALID_ARG, "h, lm_head and g_final must be 16-byte aligned");
    if (hidden < 8 || hidden % 8 || vocab < kTopK || topk < 1 || topk > kTopK || !(rms_eps >= 0.f))
        return reject(PRISM_ERR_SHAPE, "hidden must be a positive multiple of 8, vocab >= 8, topk in [1, 8]");
    if (batch < 1) return reject(PRISM_ERR_SHAPE, "batch must be >= 1");
    if (batch > kStaticMaxRows)
        return reject(PRISM_ERR_CAPACITY, "batch " + std::to_string(batch) + " exceeds the static scratch limit of " +
                                              std::to_string(kStaticMaxRows) + " rows; split the call");

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return reject(PRISM_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices) return reject(PRISM_ERR_CAPACITY, "device ordinal beyond the static setup table");
    {
        const void *ptrs[] = {h, g_final, lm_head, draft, topk_ids, topk_logits, logits, dev_flags};
        const char *names[] = {"h", "g_final", "lm_head", "draft", "topk_ids", "topk_logits", "logits", "dev_flags"};
        for (int i = 0; i < 8; ++i)
            if (!on_device(ptrs[i], dev))
                return reject(PRISM_ERR_INVALID_ARG, std::string(names[i]) + " is not device memory of the current device " +
                                                         std::to_string(dev));
    }
    DeviceState st;
    prism_status ps = setup_device(dev, st);
    if (ps != PRISM_OK) return ps;

    const bool bf16 = dtype == PRISM_BF16;
    int grid = st.sms < vocab ? st.sms : vocab;
    if (grid > kStaticMaxGrid) grid = kStaticMaxGrid;
    int *err = (int *)st.scratch;
    int *ticket = (int *)(st.scratch + 64);

    GemvArgs g{};
    g.W = lm_head;
    g.n_units = vocab;
    g.kin = hidden;
    g.T = batch;
    g.pro = kProNorm;
    g.src = h;
    g.gain = g_final;
    g.eps = rms_eps;
    g.max_new = 1;
    g.K = 1;
    g.step = 1;
    g.vocab = vocab;
    g.d = hidden;
    g.epi = kEpiTopK;
    g.logits = logits;
    g.lm_part = (float *)(st.scratch + kHeadBytes);
    g.lm_part_id = (int *)(st.scratch + kHeadBytes + kPartBytes);
    g.counter = ticket;
    g.draft_out = draft;
    g.topk_ids = topk_ids;
    g.topk_logits = topk_logits;
    g.topk = topk;
    g.err = err;
    g.force_cuda_core = 1;
    if (!gemv_supported(g, bf16)) return reject(PRISM_ERR_SHAPE, "hidden too large for the shared-memory ring");

    cudaStream_t s = (cudaStream_t)stream;
    // a call that gave up part-way can leave the ticket or the error word set
    e = cudaMemsetAsync(st.scratch, 0, kHeadBytes, s);
    if (e == cudaSuccess) e = launch_gemv(g, bf16, grid, s, false);
    if (e == cudaSuccess && dev_flags) e = cudaMemcpyAsync(dev_flags, err, sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return reject(PRISM_ERR_CUDA, std::string("LM-head launch: ") + cudaGetErrorString(e));
    return PRISM_OK;
}
