"""gv_tat_loss (token-alignable training pass, GRIFFIN Section 4.1, Eqs. 2-5)
against the float64 oracle: predictable masks and alignment masks bit-exact,
per-step and per-sequence losses within 1e-4 of the largest magnitude."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device

pytestmark = pytest.mark.gpu

TOL = 1e-4


def _run(inp, n=None, mbar_prev="cfg", k=None):
    cfg = inp.cfg
    B, T = cfg["B"], cfg["T"]
    n = cfg["n"] if n is None else n
    k = cfg["k"] if k is None else k
    prev = (inp.mbar_prev[:n - 1].contiguous() if n > 1 else None) if mbar_prev == "cfg" else mbar_prev
    dev = inp.logits.device
    mbar = torch.full((B, T), 7, dtype=torch.uint8, device=dev)
    mask = torch.full((B, T), 7, dtype=torch.uint8, device=dev)
    ell = torch.full((B, T), -1.0, dtype=torch.float32, device=dev)
    seq = torch.full((B,), -1.0, dtype=torch.float32, device=dev)
    gv.gv_tat_loss(inp.logits, inp.tokens, inp.feat_draft, inp.feat_target, k, n, prev, mbar, mask, ell, seq)
    torch.cuda.synchronize()
    return mbar.cpu().numpy(), mask.cpu().numpy(), ell.cpu().numpy(), seq.cpu().numpy()


def _oracle(inp, n, prev, k):
    f = lambda t: t.detach().cpu().double().numpy()
    return oracle.tat_pass(f(inp.logits), inp.tokens.cpu().numpy(), f(inp.feat_draft), f(inp.feat_target), k, n,
                           None if prev is None else prev.cpu().numpy())


def _rel(a, b):
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))


@pytest.mark.parametrize("logits,feat,V,H", [("f32", "bf16", 1001, 72), ("bf16", "f32", 1001, 75),
                                             ("f32", "bf16", 1024, 64), ("bf16", "bf16", 2048, 40)])
@pytest.mark.parametrize("n", [1, 2, 3])
def test_tat_small_parity(logits, feat, V, H, n):
    cfg = dict(inputs.TAT_CONFIGS["tat_small"], logits=logits, feat=feat, V=V, H=H)
    inp = inputs.make_tat_inputs(cfg, 100 + n, device=device())
    mbar, mask, ell, seq = _run(inp, n=n)
    prev = inp.mbar_prev[:n - 1] if n > 1 else None
    ref = _oracle(inp, n, prev, cfg["k"])
    np.testing.assert_array_equal(mbar, ref["mbar"])
    np.testing.assert_array_equal(mask, ref["mask"])
    assert 0 < ref["mbar"].sum() < ref["mbar"].size      # both outcomes occur
    assert _rel(ell, ref["ell"]) <= TOL
    assert _rel(seq, ref["seq_loss"]) <= TOL


def test_tat_passes_chain():
    # Passes 1, 2, 3 with fresh logits each, every pass fed the predictable
    # masks the GPU produced in the passes before it.
    cfg = dict(inputs.TAT_CONFIGS["tat_small"], V=512, H=64)
    dev = device()
    masks = []
    for n in (1, 2, 3):
        inp = inputs.make_tat_inputs(cfg, 300 + n, device=dev)
        prev = torch.stack(masks).contiguous() if masks else None
        mbar, mask, ell, seq = _run(inp, n=n, mbar_prev=prev)
        ref = _oracle(inp, n, prev, cfg["k"])
        np.testing.assert_array_equal(mbar, ref["mbar"])
        np.testing.assert_array_equal(mask, ref["mask"])
        assert _rel(seq, ref["seq_loss"]) <= TOL
        masks.append(torch.from_numpy(mbar).to(dev))


def test_tat_k_and_ties():
    # bf16 logits on a coarse grid: many ties at the target's value; k = 1 and 5.
    cfg = dict(inputs.TAT_CONFIGS["tat_small"], V=256, H=32, logits="bf16", feat="bf16")
    inp = inputs.make_tat_inputs(cfg, 7, device=device())
    inp.logits.copy_((inp.logits.float() * 2).round().to(torch.bfloat16))
    for k in (1, 5):
        mbar, mask, ell, seq = _run(inp, n=2, k=k)
        ref = _oracle(inp, 2, inp.mbar_prev[:1], k)
        np.testing.assert_array_equal(mbar, ref["mbar"])
        assert _rel(ell, ref["ell"]) <= TOL


def test_tat_bad_token_is_loud():
    cfg = dict(inputs.TAT_CONFIGS["tat_small"], V=1024, H=64)
    inp = inputs.make_tat_inputs(cfg, 9, device=device())
    inp.tokens[0, 5] = cfg["V"]
    mbar, mask, ell, seq = _run(inp, n=1)
    assert np.isnan(ell[0, 5]) and mbar[0, 5] == 0
    assert np.isnan(seq[0]) and np.isfinite(seq[1])


def test_tat_fullsize_sampled():
    # The benchmark workload (4 x 2048 positions, vocabulary 32000, hidden
    # 4096, pass 3): masks exact everywhere (the alignment mask is index
    # logic), losses on sampled rows, and the per-sequence reduction of the
    # GPU's own per-step losses.
    cfg = inputs.TAT_CONFIGS["tat_llama2_7b"]
    inp = inputs.make_tat_inputs(cfg, 1000, device=device())
    B, T = cfg["B"], cfg["T"]
    mbar, mask, ell, seq = _run(inp)
    prev = inp.mbar_prev.cpu().numpy()
    np.testing.assert_array_equal(mask, oracle.alignment_mask(prev, cfg["n"], B, T))
    rng = np.random.default_rng(0)
    rows = rng.choice(B * T, size=48, replace=False)
    lg = inp.logits.view(B * T, -1)[torch.as_tensor(rows, device=inp.logits.device)].cpu().double().numpy()
    tok = inp.tokens.view(-1).cpu().numpy()[rows]
    fd = inp.feat_draft.view(B * T, -1)[torch.as_tensor(rows, device=inp.logits.device)].cpu().double().numpy()
    ft = inp.feat_target.view(B * T, -1)[torch.as_tensor(rows, device=inp.logits.device)].cpu().double().numpy()
    np.testing.assert_array_equal(mbar.reshape(-1)[rows], oracle.predictable_mask(lg, tok, cfg["k"]))
    ref_ell = oracle.token_loss(lg, tok) + 0.1 * oracle.feature_loss(fd, ft)
    assert _rel(ell.reshape(-1)[rows], ref_ell) <= TOL
    m = mask.astype(np.float64)
    ref_seq = (m * ell).sum(axis=1) / m.sum(axis=1)
    assert _rel(seq, ref_seq) <= TOL
