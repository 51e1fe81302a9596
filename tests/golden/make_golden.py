"""Write tests/golden/tiny_rounds.json: oracle outputs on the tiny workloads.

Calls only the oracle and the seeded input generator.  Run from the
repository root:  python tests/golden/make_golden.py
"""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402


def main():
    out = {}
    for name in ("tiny-f32", "tiny-bf16", "tiny-f32-decode"):
        w = synth.WORKLOADS[name]
        W, I = synth.make_weights(w), synth.make_round_inputs(w)
        r = oracle.draft_round(w.shape, W, I, topk=4, want_logits=True)
        out[name] = {
            "draft_ids": r["draft_ids"].tolist(),
            "topk_ids": r["topk_ids"].tolist(),
            "topk_logits": r["topk_logits"].tolist(),
            "hidden_head": r["hidden_out"][:, :, :8].tolist(),
        }
    path = os.path.join(ROOT, "tests", "golden", "tiny_rounds.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
    print("wrote", path)


if __name__ == "__main__":
    main()
