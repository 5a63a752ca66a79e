"""gv_rmsnorm and gv_linear (the target layer's norms and projections around
the tree attention) against the float64 oracle, on the shapes of the verify
step (60 node rows, hidden 4096, FFN 14336) and on ragged ones (one row, two
M tiles, K not a multiple of 64, an output width that leaves a partial tile).
bf16 outputs: within 1e-2 of the largest magnitude (one bf16 rounding of an
fp32 result)."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv
from gpu_util import device, f64, rel_err

pytestmark = pytest.mark.gpu

TOL = 1e-2


def _bf(shape, gen, scale=1.0):
    return (torch.randn(shape, generator=gen) * scale).to(torch.bfloat16)


@pytest.mark.parametrize("rows,H", [(60, 4096), (7, 72), (256, 5120)])
def test_rmsnorm_parity(rows, H):
    dev = device()
    gen = torch.Generator().manual_seed(rows + H)
    x = _bf((rows, H), gen, 3.0)
    w = _bf((H,), gen)
    out = torch.empty(rows, H, dtype=torch.bfloat16, device=dev)
    gv.gv_rmsnorm(x.to(dev), w.to(dev), out, eps=1e-5)
    torch.cuda.synchronize()
    ref = oracle.rmsnorm(f64(x), f64(w), 1e-5)
    assert rel_err(f64(out), ref) <= TOL


def _linear(x, W, n_out, epi, residual=None):
    dev = device()
    rows, K = x.shape
    ws = torch.empty(gv.gv_linear_workspace(rows, K, n_out, epi), dtype=torch.uint8, device=dev)
    out = residual if residual is not None else torch.empty(rows, n_out, dtype=torch.bfloat16, device=dev)
    gv.gv_linear(x, W, out, epi, residual=residual, workspace=ws)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("rows,K,N", [(60, 4096, 4096), (60, 4096, 1024), (1, 4096, 4096), (130, 1000, 200),
                                      (256, 512, 4104), (60, 14336, 4096), (60, 4096, 28672)])
def test_linear_store_parity(rows, K, N):
    dev = device()
    gen = torch.Generator().manual_seed(rows * 7 + K + N)
    x = _bf((rows, K), gen).to(dev)
    W = _bf((N, K), gen, 0.02).to(dev)
    out = _linear(x, W, N, gv.GV_LINEAR_STORE)
    ref = oracle.linear(f64(x), f64(W))
    assert np.isfinite(f64(out)).all()
    assert rel_err(f64(out), ref) <= TOL


def test_linear_residual_in_place():
    dev = device()
    gen = torch.Generator().manual_seed(5)
    rows, K, N = 60, 4096, 4096
    x = _bf((rows, K), gen).to(dev)
    W = _bf((N, K), gen, 0.02).to(dev)
    h = _bf((rows, N), gen, 2.0).to(dev)
    h0 = f64(h)
    _linear(x, W, N, gv.GV_LINEAR_ADD, residual=h)     # h += x W^T, in place
    ref = h0 + oracle.linear(f64(x), f64(W))
    assert rel_err(f64(h), ref) <= TOL


@pytest.mark.parametrize("rows,K,F", [(60, 4096, 14336), (9, 256, 520)])
def test_linear_swiglu_parity(rows, K, F):
    dev = device()
    gen = torch.Generator().manual_seed(rows + F)
    x = _bf((rows, K), gen).to(dev)
    Wg = _bf((F, K), gen, 0.02)
    Wu = _bf((F, K), gen, 0.02)
    W = torch.cat([Wg, Wu], 0).contiguous().to(dev)
    out = _linear(x, W, F, gv.GV_LINEAR_SWIGLU)
    ref = oracle.swiglu(f64(x), f64(Wg), f64(Wu))
    assert rel_err(f64(out), ref) <= TOL


def test_linear_workspace_reuse_dirty():
    # The workspace holds only this call's partial sums: a dirty buffer and
    # back-to-back calls of different shapes give the same results.
    dev = device()
    gen = torch.Generator().manual_seed(11)
    shapes = [(1024, 4096), (4096, 14336), (1024, 4096)]
    size = max(gv.gv_linear_workspace(60, K, N, gv.GV_LINEAR_STORE) for N, K in shapes)
    ws = torch.full((size,), 0xFF, dtype=torch.uint8, device=dev)
    outs = []
    for (N, K) in shapes:
        x = _bf((60, K), torch.Generator().manual_seed(K)).to(dev)
        W = _bf((N, K), torch.Generator().manual_seed(N + K), 0.02).to(dev)
        out = torch.empty(60, N, dtype=torch.bfloat16, device=dev)
        gv.gv_linear(x, W, out, gv.GV_LINEAR_STORE, workspace=ws)
        torch.cuda.synchronize()
        assert rel_err(f64(out), oracle.linear(f64(x), f64(W))) <= TOL
        outs.append(out.clone())
    assert torch.equal(outs[0], outs[2])


@pytest.mark.parametrize("rows,K,nq,nkv", [(60, 4096, 4096, 1024), (240, 5120, 5120, 5120), (5, 256, 64, 32)])
def test_linear_qkv_parity(rows, K, nq, nkv):
    dev = device()
    gen = torch.Generator().manual_seed(rows + nq + nkv)
    x = _bf((rows, K), gen).to(dev)
    W = _bf((nq + 2 * nkv, K), gen, 0.02).to(dev)
    q = torch.empty(rows, nq, dtype=torch.bfloat16, device=dev)
    k = torch.empty(rows, nkv, dtype=torch.bfloat16, device=dev)
    v = torch.empty(rows, nkv, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(gv.gv_linear_qkv_workspace(rows, K, nq, nkv), dtype=torch.uint8, device=dev)
    gv.gv_linear_qkv(x, W, q, k, v, ws)
    torch.cuda.synchronize()
    ref = oracle.linear(f64(x), f64(W))
    assert rel_err(f64(q), ref[:, :nq]) <= TOL
    assert rel_err(f64(k), ref[:, nq:nq + nkv]) <= TOL
    assert rel_err(f64(v), ref[:, nq + nkv:]) <= TOL


@pytest.mark.parametrize("rows,K,N", [(60, 4096, 4096), (240, 13824, 5120), (3, 64, 40)])
def test_linear_add_rmsnorm_parity(rows, K, N):
    dev = device()
    gen = torch.Generator().manual_seed(rows + K)
    x = _bf((rows, K), gen).to(dev)
    W = _bf((N, K), gen, 0.02).to(dev)
    h = _bf((rows, N), gen, 2.0).to(dev)
    g = _bf((N,), gen).to(dev)
    h0 = f64(h)
    xn = torch.empty(rows, N, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(gv.gv_linear_workspace(rows, K, N, gv.GV_LINEAR_ADD), dtype=torch.uint8, device=dev)
    gv.gv_linear_add_rmsnorm(x, W, h, h, g, xn, ws)      # in place on h
    torch.cuda.synchronize()
    ref_h = h0 + oracle.linear(f64(x), f64(W))
    assert rel_err(f64(h), ref_h) <= TOL
    # the norm is taken of the stored (rounded) h
    assert rel_err(f64(xn), oracle.rmsnorm(f64(h), f64(g), 1e-5)) <= TOL
