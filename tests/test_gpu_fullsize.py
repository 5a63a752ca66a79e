"""Full-size parity: the whole benchmark step -- every layer, the benchmark
seed, the CUDA graph bench.py replays -- on the LLaMA-3-8B workload (32
layers, prefix 4096, vocabulary 128256, greedy; the benchmark's own
workload), the LLaMA-2-7B and the batch-4 LLaMA-2-13B workloads (greedy; the
latter with ragged prefixes up to 8192 and more CTAs than SMs), and the
Mixtral-attention workload (32 layers, prefix 16384, temperature 1).

The float64 oracle cannot redo all 32 layers in seconds, so it checks samples
that it can compute one by one: the first, a middle and the last layer's
attention output and tree keys/values over every head, every layer's over one
KV-head group (group l mod Hkv, so a wrong layer or head offset anywhere in
the multi-layer call shows); the LM-head argmax of a sample of rows
(every row's argmax is also checked against the planted closed form); the
acceptance of the GPU's choices (bit-exact for greedy, a valid trail under the
oracle's probabilities for sampling); the compacted rows of the sampled
layers, and sampled cache rows that must not change."""

import numpy as np
import pytest
import torch

import oracle
from oracle.accept import check_sampling_trail
from paper_2502_11018_gb300 import inputs
from paper_2502_11018_gb300.step import VerifyStep
from gpu_util import device, f64, rel_err, TOL_ATTN, TOL_ROT

pytestmark = pytest.mark.gpu

BENCH_SEED = 1000   # bench.py's default seed (rank 0)


def _run_bench_step(name):
    dev = device()
    cfg = inputs.config(name)
    inp = inputs.make_step_inputs(cfg, BENCH_SEED, device=dev)
    L = cfg["L"]
    layers = sorted({0, L // 2, L - 1})
    P = inp.prefix_len.cpu().numpy()
    D = cfg["D"]
    # Cache rows the step may write (P .. P + D) and a few it must not touch,
    # before the step runs.
    keep = {l: (inp.cacheK[l].cpu().clone(), inp.cacheV[l].cpu().clone()) for l in layers}
    step = VerifyStep(inp)
    step.capture()
    step.replay()
    torch.cuda.synchronize()
    return cfg, inp, step, layers, keep, P, D


def _check_tree_attention_compaction(cfg, inp, step, layers, keep, P):
    parents = inp.parents.cpu().numpy()
    depth, pos, anc, st = oracle.tree_build(parents, P)
    np.testing.assert_array_equal(step.depth.cpu().numpy(), depth)
    np.testing.assert_array_equal(step.pos.cpu().numpy(), pos)
    np.testing.assert_array_equal(step.anc.cpu().numpy().view(np.uint64), anc)
    kind = cfg["dtype"]
    for l in layers:
        cK, cV = keep[l]
        ro, rK, rV = oracle.tree_attention(f64(inp.q[l]), f64(inp.k_new[l]), f64(inp.v_new[l]),
                                           f64(cK), f64(cV), P, pos, anc, cfg["rope_base"])
        out = f64(step.attn_out[l])
        assert np.isfinite(out).all()
        assert rel_err(out, ro) <= TOL_ATTN[kind], l
        assert rel_err(f64(step.treeK[l]), rK) <= TOL_ROT[kind], l
        np.testing.assert_array_equal(f64(step.treeV[l]), rV)
    # Every layer, one KV-head group each (the query heads g G .. g G + G - 1
    # that share KV head g).  The prefix rows read here are the cache's rows
    # below P, which the compaction never writes.
    Hkv = cfg["Hkv"]
    G = cfg["Hq"] // Hkv
    for l in range(cfg["L"]):
        g = l % Hkv
        hs = slice(g * G, (g + 1) * G)
        gs = slice(g, g + 1)
        ro, rK, rV = oracle.tree_attention(f64(inp.q[l][:, :, hs]), f64(inp.k_new[l][:, :, gs]),
                                           f64(inp.v_new[l][:, :, gs]), f64(inp.cacheK[l][:, gs]),
                                           f64(inp.cacheV[l][:, gs]), P, pos, anc, cfg["rope_base"])
        out = f64(step.attn_out[l][:, :, hs])
        assert np.isfinite(out).all(), (l, g)
        assert rel_err(out, ro) <= TOL_ATTN[kind], (l, g)
        assert rel_err(f64(step.treeK[l][:, gs]), rK) <= TOL_ROT[kind], (l, g)
        np.testing.assert_array_equal(f64(step.treeV[l][:, gs]), rV)
    # Compaction of the sampled layers: accepted rows come from the tree
    # scratch, every other row keeps its bytes.
    path = step.path.cpu().numpy()
    alen = step.accept_len.cpu().numpy()
    np.testing.assert_array_equal(step.new_len.cpu().numpy(), P + alen)
    for l in layers:
        gK, gV = inp.cacheK[l].cpu(), inp.cacheV[l].cpu()
        tK, tV = step.treeK[l].cpu(), step.treeV[l].cpu()
        cK, cV = keep[l]
        for b in range(cfg["B"]):
            lo, hi = int(P[b]), int(P[b] + alen[b])
            for t in range(alen[b]):
                assert torch.equal(gK[b, :, lo + t], tK[b, :, path[b, t]])
                assert torch.equal(gV[b, :, lo + t], tV[b, :, path[b, t]])
            for r in (0, lo // 2, lo - 1, hi, cfg["S_max"] - 1):
                if 0 <= r < lo or hi <= r < cfg["S_max"]:
                    assert torch.equal(gK[b, :, r], cK[b, :, r]) and torch.equal(gV[b, :, r], cV[b, :, r])
    return parents, path, alen


@pytest.mark.parametrize("name", ["llama3_8b", "llama2_7b", "llama2_13b_b4"])
def test_fullsize_greedy(name):
    cfg, inp, step, layers, keep, P, D = _run_bench_step(name)
    parents, path, alen = _check_tree_attention_compaction(cfg, inp, step, layers, keep, P)
    ids = step.ids.cpu().numpy()
    # Every row's argmax is the planted token (margin > 1 by construction) ...
    np.testing.assert_array_equal(ids, inp.planted.cpu().numpy().reshape(-1))
    # ... and, on a sample of rows, the float64 LM head's argmax.
    rows = sorted({0, 1, 17, 31, 45, ids.size // 2, ids.size - 1})
    h = f64(inp.h)[rows]
    W = f64(inp.W)
    ref_ids, _ = oracle.select_argmax(oracle.lmhead_logits(h, W))
    np.testing.assert_array_equal(ids[rows], ref_ids)
    tokens = inp.tokens.cpu().numpy()
    rpath, rlen, rout, rst = oracle.accept_greedy(parents, tokens, ids, D)
    np.testing.assert_array_equal(path, rpath)
    np.testing.assert_array_equal(alen, rlen)
    np.testing.assert_array_equal(step.out_tokens.cpu().numpy(), rout)
    assert (step.seq_status.cpu().numpy() == 0).all()


def test_fullsize_mixtral_sampling():
    cfg, inp, step, layers, keep, P, D = _run_bench_step("mixtral_attn")
    parents, path, alen = _check_tree_attention_compaction(cfg, inp, step, layers, keep, P)
    B, N = cfg["B"], cfg["N"]
    tl = oracle.lmhead_logits(f64(inp.h), f64(inp.W)).reshape(B, N, -1)
    # The GPU's fp32 logits, row max and log-sum-exp against float64.
    assert rel_err(f64(step.logits).reshape(B, N, -1), tl) <= 1e-3
    tokens = inp.tokens.cpu().numpy()
    out = step.out_tokens.cpu().numpy()
    for b in range(B):
        trail = path[b, :alen[b]].tolist()
        ok, _ = check_sampling_trail(parents[b], tokens[b], tl[b], f64(inp.draft_logits[b]),
                                     f64(inp.u_acc[b]), f64(inp.u_res[b]), trail,
                                     int(out[b, alen[b] - 1]), cfg["temperature"], tol=1e-4)
        assert ok, trail
    assert (step.seq_status.cpu().numpy() == 0).all()
