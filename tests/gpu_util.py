"""Helpers shared by the GPU parity tests (test infrastructure)."""

import numpy as np
import torch

from paper_2502_11018_gb300 import build

_built = False


def device():
    """Build libgv.so once per session and return the CUDA device.

    A GPU test must never pass on a silent fallback, so a missing GPU is an
    error here, not a skip.
    """
    global _built
    if not _built:
        build.build()
        _built = True
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda", 0)


def f64(t):
    return t.detach().cpu().double().numpy()


def rel_err(got, ref):
    """max |got - ref| / max |ref| (the tolerance measure of every float check)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    scale = np.abs(ref).max()
    return float(np.abs(got - ref).max() / (scale if scale > 0 else 1.0))


# Tolerances, relative to the largest oracle magnitude of the compared tensor.
# Attention outputs: the stated 2e-2 (bf16 operands, bf16 output) and 1e-4
# (fp32).  bf16 rounding of one value is 2^-9 relative, so rotated tree keys
# are held to 1e-2 (bf16) / 1e-5 (fp32).
TOL_ATTN = {"bf16": 2e-2, "f32": 1e-4}
TOL_ROT = {"bf16": 1e-2, "f32": 1e-5}
# Logits accumulate exact bf16 products in fp32 over H <= 8192 terms.
TOL_LOGITS = {"bf16": 1e-3, "f32": 1e-5}


def to_device(inp, dev):
    """Copy every tensor field of a StepInputs to ``dev`` (returns a new object)."""
    import dataclasses
    kw = {}
    for f in dataclasses.fields(inp):
        v = getattr(inp, f.name)
        kw[f.name] = v.to(dev) if isinstance(v, torch.Tensor) else v
    return type(inp)(**kw)
