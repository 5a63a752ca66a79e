"""gv_tgf (the draft model's Token-Guided Fusion, Eqs. 6-8) through the C
ABI against the float64 oracle.  h is one bf16 rounding of an fp32 sum (held
to 1e-2 of its largest magnitude); o follows three projections with bf16
roundings of h, the normalised input and silu(z) in between, each a relative
2^-9 that the next projection averages over thousands of terms: 2e-2."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device, f64, rel_err

pytestmark = pytest.mark.gpu

TOL_H = 1e-2
TOL_O = 2e-2


def _run(ti, ws=None):
    dev = ti.F.device
    rows, d = ti.F.shape
    e = ti.w["Wu"].shape[0]
    h = torch.empty(rows, d, dtype=torch.bfloat16, device=dev)
    o = torch.empty(rows, d, dtype=torch.bfloat16, device=dev)
    if ws is None:
        ws = torch.empty(gv.gv_tgf_workspace(rows, d, e), dtype=torch.uint8, device=dev)
    gv.gv_tgf(ti.F, ti.x, ti.w, h, o, ws)
    torch.cuda.synchronize()
    return h, o


def _oracle(ti):
    w = {k: f64(v) for k, v in ti.w.items()}
    return oracle.tgf_forward(f64(ti.F), f64(ti.x), w)


@pytest.mark.parametrize("name,over", [
    ("tgf_small", {}),
    ("tgf_small", dict(rows=1, d=64, e=72)),
    ("tgf_llama2_7b", {}),
    ("tgf_llama2_7b_r256", {}),
    ("tgf_llama2_7b", dict(rows=33, d=8192, e=4096)),
])
def test_tgf_parity(name, over):
    cfg = dict(inputs.TGF_CONFIGS[name], **over)
    ti = inputs.make_tgf_inputs(cfg, 7, device=device())
    h, o = _run(ti)
    ref_o, ref_h = _oracle(ti)
    assert np.isfinite(f64(o)).all()
    assert rel_err(f64(h), ref_h) <= TOL_H
    assert rel_err(f64(o), ref_o) <= TOL_O


def test_tgf_dirty_workspace_and_graph_replay():
    # The workspace holds only this call's scratch: a 0xFF-filled buffer, a
    # second call and a CUDA-graph replay give bit-identical outputs.
    cfg = inputs.TGF_CONFIGS["tgf_small"]
    ti = inputs.make_tgf_inputs(cfg, 3, device=device())
    rows, d, e = cfg["rows"], cfg["d"], cfg["e"]
    ws = torch.full((gv.gv_tgf_workspace(rows, d, e),), 0xFF, dtype=torch.uint8, device=device())
    h0, o0 = _run(ti, ws)
    h1, o1 = _run(ti, ws)
    assert torch.equal(h0, h1) and torch.equal(o0, o1)
    h = torch.zeros_like(h0)
    o = torch.zeros_like(o0)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        gv.gv_tgf(ti.F, ti.x, ti.w, h, o, ws, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        gv.gv_tgf(ti.F, ti.x, ti.w, h, o, ws, stream=torch.cuda.current_stream())
    h.zero_()
    o.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(h, h0) and torch.equal(o, o0)


def test_linear_silu_bias_free_parity():
    # the public SiLU epilogue of gv_linear (the Up Projector's activation)
    dev = device()
    gen = torch.Generator().manual_seed(9)
    x = (torch.randn(60, 1024, generator=gen)).to(torch.bfloat16).to(dev)
    W = (torch.randn(2056, 1024, generator=gen) * 0.02).to(torch.bfloat16).to(dev)
    out = torch.empty(60, 2056, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(gv.gv_linear_workspace(60, 1024, 2056, gv.GV_LINEAR_SILU), dtype=torch.uint8, device=dev)
    gv.gv_linear(x, W, out, gv.GV_LINEAR_SILU, workspace=ws)
    torch.cuda.synchronize()
    assert rel_err(f64(out), oracle.silu(oracle.linear(f64(x), f64(W)))) <= 1e-2
