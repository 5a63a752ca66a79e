"""GPU parity of gv_verify_attention_layers (the attention of L layers in one
persistent launch) against the float64 oracle, layer by layer.

The cases cover the ways the launch cuts its work: one or two 128-row query
tiles per KV head (MHA, GQA with G * N up to 256), ragged batches with empty
and one-key prefixes, fewer blocks than CTAs (most CTAs idle), a single unit
cut into pieces across every CTA (the last piece to arrive merges up to one
piece per SM), units cut at range ends, strided layer inputs (views of a
packed per-layer buffer) and a workspace that starts dirty and is reused.
Tolerances as for gv_verify_attention: output 2e-2 of its largest magnitude,
rotated tree keys 1e-2, tree values exact."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device, f64, rel_err, TOL_ATTN, TOL_ROT

pytestmark = pytest.mark.gpu

CASES = [
    # L, B, N, Hq, Hkv, prefixes, rope base
    (3, 1, 60, 32, 8, [300], 5e5),                   # LLaMA-3-8B heads: two tiles per KV head
    (2, 1, 60, 32, 8, [4096], 5e5),                  # the benchmark's prefix
    (2, 2, 60, 8, 8, [129, 2100], 1e4),              # MHA: one tile
    (2, 3, 64, 8, 2, [0, 1, 1000], 1e6),             # 256 rows per KV head, empty prefix
    (1, 1, 1, 2, 2, [0], 1e4),                       # one block in all: 151 idle CTAs
    (3, 2, 17, 4, 4, [127, 128], 1e4),
    (1, 1, 60, 4, 1, [25600], 1e4),                  # one unit cut across every CTA
    (2, 1, 61, 16, 4, [777], 5e5),                   # 244 rows per KV head
    (2, 16, 3, 32, 8, [512, 768, 1024, 1536] * 4, 5e5),   # batched chains
    (2, 4, 60, 40, 40, [64, 65, 255, 256], 1e4),     # ragged batch, MHA
    (1, 64, 4, 8, 8, [(37 * i) % 600 for i in range(64)], 1e4),   # 64 sequences, the most a call takes
    (2, 2, 40, 12, 4, [333, 0], 5e5),                # G = 3: 42 nodes per 128-row tile, 120 rows
]


def _case(L, B, N, Hq, Hkv, P, seed):
    rng = np.random.default_rng(seed)
    gen = torch.Generator().manual_seed(seed)
    parents = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        parents[b] = [-1] if N == 1 else inputs.make_tree(rng, N, min(8, N - 1), 10, 100)[0]
    S_max = max(P) + 70
    bf = torch.bfloat16
    q = torch.randn(L, B, N, Hq, 128, generator=gen).to(bf)
    k = torch.randn(L, B, N, Hkv, 128, generator=gen).to(bf)
    v = torch.randn(L, B, N, Hkv, 128, generator=gen).to(bf)
    cK = torch.randn(L, B, Hkv, S_max, 128, generator=gen).to(bf)
    cV = torch.randn(L, B, Hkv, S_max, 128, generator=gen).to(bf)
    return parents, np.array(P, dtype=np.int32), S_max, q, k, v, cK, cV


def _tree(dev, parents, P, base, d=128):
    B, N = parents.shape
    t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    depth = torch.zeros(B, N, dtype=torch.int32, device=dev)
    pos = torch.zeros_like(depth)
    anc = torch.zeros(B, N, dtype=torch.int64, device=dev)
    st = torch.zeros(B, dtype=torch.int32, device=dev)
    Pd = t(P)
    gv.gv_tree_build(t(parents), Pd, depth, pos, anc, st)
    rope = torch.zeros(B, N, d // 2, 2, dtype=torch.float32, device=dev)
    gv.gv_rope_table(pos, d, base, rope)
    return Pd, rope, anc


def run_layers(dev, parents, P, S_max, q, k, v, cK, cV, base, ws=None):
    L, B, N, Hq, _ = q.shape
    Hkv = k.shape[3]
    Pd, rope, anc = _tree(dev, parents, P, base)
    shape = gv.attn_shape(B, N, Hq, Hkv, 128, S_max, gv.GV_BF16)
    if ws is None:
        ws = torch.full((gv.gv_verify_attention_layers_workspace(shape, L),), 0xFF, dtype=torch.uint8, device=dev)
    tK = torch.zeros(L, B, Hkv, N, 128, dtype=torch.bfloat16, device=dev)
    tV = torch.zeros_like(tK)
    out = torch.zeros(L, B, N, Hq, 128, dtype=torch.bfloat16, device=dev)
    gv.gv_verify_attention_layers(shape, q.to(dev), k.to(dev), v.to(dev), cK.to(dev), cV.to(dev), Pd, rope, anc,
                                  tK, tV, out, ws)
    torch.cuda.synchronize()
    return out, tK, tV


def oracle_layers(parents, P, q, k, v, cK, cV, base):
    """The float64 oracle's (out, tree K, tree V) of every layer."""
    depth, pos, anc, _ = oracle.tree_build(parents, P)
    return [oracle.tree_attention(f64(q[l]), f64(k[l]), f64(v[l]), f64(cK[l]), f64(cV[l]), P, pos, anc, base)
            for l in range(q.shape[0])]


def check_layers(out, tK, tV, parents, P, q, k, v, cK, cV, base, refs=None):
    refs = refs if refs is not None else oracle_layers(parents, P, q, k, v, cK, cV, base)
    for l in range(q.shape[0]):
        ro, rK, rV = refs[l]
        o = f64(out[l])
        assert np.isfinite(o).all(), l
        assert rel_err(o, ro) <= TOL_ATTN["bf16"], (l, rel_err(o, ro))
        assert rel_err(f64(tK[l]), rK) <= TOL_ROT["bf16"], l
        np.testing.assert_array_equal(f64(tV[l]), rV)


@pytest.mark.parametrize("case", range(len(CASES)))
def test_attention_layers_parity(case):
    dev = device()
    L, B, N, Hq, Hkv, P, base = CASES[case]
    parents, P, S_max, q, k, v, cK, cV = _case(L, B, N, Hq, Hkv, P, 300 + case)
    out, tK, tV = run_layers(dev, parents, P, S_max, q, k, v, cK, cV, base)
    check_layers(out, tK, tV, parents, P, q, k, v, cK, cV, base)


def test_attention_layers_matches_per_layer_calls():
    """Every layer against gv_verify_attention on the same inputs: the tree
    K/V scratch bit for bit, the outputs within the tolerance (the two calls
    cut the keys differently, so the last bf16 bit may differ)."""
    dev = device()
    L, B, N, Hq, Hkv, P, base = 3, 2, 60, 32, 8, [700, 1500], 5e5
    parents, P, S_max, q, k, v, cK, cV = _case(L, B, N, Hq, Hkv, P, 21)
    out, tK, tV = run_layers(dev, parents, P, S_max, q, k, v, cK, cV, base)
    Pd, rope, anc = _tree(dev, parents, P, base)
    shape = gv.attn_shape(B, N, Hq, Hkv, 128, S_max, gv.GV_BF16)
    ws = torch.empty(gv.gv_verify_attention_workspace(shape), dtype=torch.uint8, device=dev)
    for l in range(L):
        tK1 = torch.zeros(B, Hkv, N, 128, dtype=torch.bfloat16, device=dev)
        tV1 = torch.zeros_like(tK1)
        o1 = torch.zeros(B, N, Hq, 128, dtype=torch.bfloat16, device=dev)
        gv.gv_verify_attention(shape, q[l].to(dev), k[l].to(dev), v[l].to(dev), cK[l].to(dev), cV[l].to(dev), Pd,
                               rope, anc, tK1, tV1, o1, ws)
        torch.cuda.synchronize()
        assert torch.equal(tK1, tK[l]) and torch.equal(tV1, tV[l])
        assert rel_err(f64(out[l]), f64(o1)) <= TOL_ATTN["bf16"]


def test_attention_layers_reused_workspace_and_strided_layers():
    """Eight calls on one dirty workspace: the tree K/V scratch agrees bit for
    bit, and every call's outputs pass the float64 oracle's bound and agree
    with the first call's to 2^-6 of their scale.  (A unit cut between two
    CTAs is combined by whichever of its pieces arrives second, from its fp32
    accumulators and the other's bf16 partial rows, or merged from both
    partials when they arrive together: equally valid roundings, so calls
    need not agree bit for bit.)  Inputs given as views of a packed per-layer
    buffer (q | k_new | v_new per layer) give the same tree K/V bits."""
    dev = device()
    L, B, N, Hq, Hkv, P, base = 4, 2, 60, 32, 8, [1000, 3000], 5e5
    parents, P, S_max, q, k, v, cK, cV = _case(L, B, N, Hq, Hkv, P, 22)
    shape = gv.attn_shape(B, N, Hq, Hkv, 128, S_max, gv.GV_BF16)
    ws = torch.full((gv.gv_verify_attention_layers_workspace(shape, L),), 0xFF, dtype=torch.uint8, device=dev)
    outs = [run_layers(dev, parents, P, S_max, q, k, v, cK, cV, base, ws) for _ in range(8)]
    for o in outs[1:]:
        assert torch.equal(o[1], outs[0][1]) and torch.equal(o[2], outs[0][2])
        assert rel_err(f64(o[0]), f64(outs[0][0])) <= 2.0 ** -6
    refs = oracle_layers(parents, P, q, k, v, cK, cV, base)
    for o in outs:
        check_layers(o[0], o[1], o[2], parents, P, q, k, v, cK, cV, base, refs)
    nq, nk = q[0].numel(), k[0].numel()
    packed = torch.empty(L, nq + 2 * nk, dtype=torch.bfloat16, device=dev)
    packed[:, :nq] = q.reshape(L, nq).to(dev)
    packed[:, nq:nq + nk] = k.reshape(L, nk).to(dev)
    packed[:, nq + nk:] = v.reshape(L, nk).to(dev)
    qv = packed[:, :nq].view(q.shape)
    kv = packed[:, nq:nq + nk].view(k.shape)
    vv = packed[:, nq + nk:].view(v.shape)
    Pd, rope, anc = _tree(dev, parents, P, base)
    tK = torch.zeros(L, B, Hkv, N, 128, dtype=torch.bfloat16, device=dev)
    tV = torch.zeros_like(tK)
    out = torch.zeros(L, B, N, Hq, 128, dtype=torch.bfloat16, device=dev)
    gv.gv_verify_attention_layers(shape, qv, kv, vv, cK.to(dev), cV.to(dev), Pd, rope, anc, tK, tV, out, ws)
    torch.cuda.synchronize()
    assert torch.equal(tK, outs[0][1]) and torch.equal(tV, outs[0][2])
    assert rel_err(f64(out), f64(outs[0][0])) <= 2.0 ** -6
