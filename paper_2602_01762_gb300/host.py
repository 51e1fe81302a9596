"""Host-side marshalling helpers: move numpy arrays (bf16 kept as uint16 bit
patterns) to device tensors and bind a drafter's weights."""
from __future__ import annotations

import numpy as np
import torch

from . import STEP_TENSORS, Drafter


def to_device(a: np.ndarray, device="cuda", pin=False) -> torch.Tensor:
    """uint16 arrays are bf16 bit patterns; others keep their dtype."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        t = torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(a)
    if pin:
        t = t.pin_memory()
    return t.to(device, non_blocking=pin)


def to_numpy(t: torch.Tensor) -> np.ndarray:
    """Inverse of to_device (bf16 -> uint16 bit patterns)."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def bind_weights(drafter: Drafter, weights: dict, device="cuda") -> dict:
    """Upload embedding, LM head and every module once; bind step k to module
    f_map[k] (steps that share a module share its device tensors)."""
    dev = {"embed": to_device(weights["embed"], device), "lm_head": to_device(weights["lm_head"], device),
           "modules": {}}
    for m, mod in weights["modules"].items():
        dev["modules"][m] = {n: to_device(mod[n], device) for n in STEP_TENSORS}
    drafter.load_shared_weights(dev["embed"], dev["lm_head"])
    for k, m in enumerate(weights["f_map"]):
        drafter.load_step_weights(k, dev["modules"][m])
    return dev
