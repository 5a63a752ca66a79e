"""GPU parity of gv_lmhead_select against the float64 oracle.

argmax ids are compared bit-exactly: hidden states are planted so that the
planted token beats every other score by a margin far above the arithmetic
error.  Top-k ids are compared exactly wherever consecutive oracle scores are
separated by more than the tolerance, and the values everywhere.  Logits and
log-sum-exp are compared within 1e-3 (bf16) / 1e-5 (fp32) of the largest
magnitude."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device, f64, rel_err, TOL_LOGITS

pytestmark = pytest.mark.gpu

CASES = [
    # dtype, rows, H, V
    ("f32", 16, 512, 4096),        # tiny workload's LM head
    ("f32", 33, 256, 1000),
    ("bf16", 60, 4096, 32000),     # LLaMA-2-7B / Mixtral vocab
    ("bf16", 1, 128, 4097),        # ragged vocab tail
    ("bf16", 240, 5120, 32000),    # 4 sequences x 60 nodes, LLaMA-2-13B hidden
    ("bf16", 61, 1024, 50000),
    # vocabulary splits of the tensor-core kernel: five tiles of 13 / 14 row
    # groups per CTA at the 64-row limit of the stage layout that lets the
    # MMA read past the hidden rows; fewer 16-row groups than CTAs; one
    # partial group
    ("bf16", 64, 256, 160000),
    ("bf16", 3, 64, 100),
    ("bf16", 2, 64, 15),
    ("bf16", 300, 128, 4097),      # two 256-row launches
]


def _inputs(dtype, rows, H, V, seed):
    gen = torch.Generator().manual_seed(seed)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    W = (torch.randn(V, H, generator=gen) * 0.02).to(dt)
    targets = torch.randint(0, V, (rows,), generator=gen)
    h = inputs.planted_hidden(gen, W, targets)
    return h, W, targets


def _oracle_logits(h, W):
    return oracle.lmhead_logits(f64(h), f64(W))


@pytest.mark.parametrize("case", range(len(CASES)))
def test_argmax_parity(case):
    dev = device()
    dtype, rows, H, V = CASES[case]
    h, W, targets = _inputs(dtype, rows, H, V, 10 + case)
    ref = _oracle_logits(h, W)
    rid, rval = oracle.select_argmax(ref)
    np.testing.assert_array_equal(rid, targets.numpy())
    ids = torch.full((rows,), -7, dtype=torch.int32, device=dev)
    vals = torch.zeros(rows, dtype=torch.float32, device=dev)
    ws = torch.empty(gv.gv_lmhead_workspace(rows, H, V, gv.dtype_code(h), gv.GV_SELECT_ARGMAX),
                     dtype=torch.uint8, device=dev)
    for _ in range(3):      # (calls reusing one workspace agree)
        ids.fill_(-7)
        gv.gv_lmhead_select(h.to(dev), W.to(dev), gv.GV_SELECT_ARGMAX, 1, ids, vals, None, None, None, ws)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(ids.cpu().numpy(), rid)
        assert rel_err(vals.cpu().numpy(), rval) <= TOL_LOGITS[dtype]


@pytest.mark.parametrize("case", [0, 2, 3, 4, 6, 7])
@pytest.mark.parametrize("k", [1, 3, 10, 16])
def test_topk_parity(case, k):
    dev = device()
    dtype, rows, H, V = CASES[case]
    h, W, targets = _inputs(dtype, rows, H, V, 20 + case)
    ref = _oracle_logits(h, W)
    rid, rval = oracle.select_topk(ref, k)
    ids = torch.zeros(rows, k, dtype=torch.int32, device=dev)
    vals = torch.zeros(rows, k, dtype=torch.float32, device=dev)
    ws = torch.empty(gv.gv_lmhead_workspace(rows, H, V, gv.dtype_code(h), gv.GV_SELECT_TOPK, k),
                     dtype=torch.uint8, device=dev)
    gv.gv_lmhead_select(h.to(dev), W.to(dev), gv.GV_SELECT_TOPK, k, ids, vals, None, None, None, ws)
    torch.cuda.synchronize()
    gi, gval = ids.cpu().numpy(), vals.cpu().numpy()
    tol = TOL_LOGITS[dtype] * np.abs(ref).max()
    assert np.abs(gval - rval).max() <= tol
    assert (np.diff(gval, axis=1) <= 0).all()
    for r in range(rows):
        for j in range(k):
            gap_prev = rval[r, j - 1] - rval[r, j] if j > 0 else np.inf
            gap_next = rval[r, j] - rval[r, j + 1] if j + 1 < k else np.inf
            if min(gap_prev, gap_next) > 2 * tol:
                assert gi[r, j] == rid[r, j], (r, j)
            # whatever id the GPU chose must carry (about) the score it reports
            assert abs(ref[r, gi[r, j]] - gval[r, j]) <= tol


@pytest.mark.parametrize("case", [0, 2, 3, 6, 7, 8])
def test_logits_lse_parity(case):
    dev = device()
    dtype, rows, H, V = CASES[case]
    h, W, _ = _inputs(dtype, rows, H, V, 30 + case)
    ref = _oracle_logits(h, W)
    rm, rlse = oracle.row_logsumexp(ref)
    logits = torch.zeros(rows, V, dtype=torch.float32, device=dev)
    rmax = torch.zeros(rows, dtype=torch.float32, device=dev)
    rl = torch.zeros(rows, dtype=torch.float32, device=dev)
    ws = torch.empty(gv.gv_lmhead_workspace(rows, H, V, gv.dtype_code(h), gv.GV_SELECT_LOGITS),
                     dtype=torch.uint8, device=dev)
    gv.gv_lmhead_select(h.to(dev), W.to(dev), gv.GV_SELECT_LOGITS, 1, None, None, logits, rmax, rl, ws)
    torch.cuda.synchronize()
    assert rel_err(logits.cpu().numpy(), ref) <= TOL_LOGITS[dtype]
    assert rel_err(rmax.cpu().numpy(), rm) <= TOL_LOGITS[dtype]
    assert np.abs(rl.cpu().numpy() - rlse).max() <= 1e-4 * max(1.0, np.abs(rlse).max())
