"""GPU parity of gv_verify_attention against the float64 oracle.

Shapes span several key tiles and splits with ragged tails (prefixes of 0,
1, 127, 128, 129, 300, 1000+ keys, cache capacities that are not tile
multiples), MHA and GQA head groups, head dims 64 and 128, trees of 1..64
nodes.  Tolerance: max |gpu - oracle| <= tol * max |oracle| per tensor, with
tol = 2e-2 (bf16) / 1e-4 (fp32) on the attention output, 1e-2 / 1e-5 on the
rotated tree keys; the tree values are a copy and must match exactly."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device, f64, rel_err, TOL_ATTN, TOL_ROT

pytestmark = pytest.mark.gpu

CASES = [
    # dtype, B, N, Hq, Hkv, d, prefixes, rope base, value std
    ("f32", 1, 16, 8, 8, 64, [256], 1e4, 0.02),        # the tiny workload's layer
    ("f32", 1, 16, 8, 8, 64, [256], 1e4, 1.0),
    ("f32", 2, 7, 4, 2, 64, [0, 129], 1e4, 1.0),
    ("f32", 2, 60, 8, 2, 128, [300, 37], 5e5, 1.0),
    ("bf16", 1, 60, 32, 8, 128, [300], 5e5, 1.0),     # LLaMA-3-8B heads, short prefix
    ("bf16", 2, 17, 4, 4, 128, [127, 128], 1e4, 1.0),
    ("bf16", 3, 64, 8, 2, 128, [1, 513, 1000], 1e6, 1.0),   # 256 query rows per KV head
    ("bf16", 1, 1, 2, 2, 128, [0], 1e4, 1.0),
    ("bf16", 2, 60, 8, 8, 128, [129, 2100], 1e4, 1.0),
    ("bf16", 1, 61, 16, 4, 128, [777], 5e5, 1.0),
    ("bf16", 4, 60, 40, 40, 128, [64, 65, 255, 256], 1e4, 1.0),  # ragged batch, MHA
    ("f32", 1, 1, 2, 2, 64, [0], 1e4, 1.0),
    ("f32", 1, 61, 16, 4, 64, [777], 5e5, 1.0),
]


def _case(dtype, B, N, Hq, Hkv, d, P, base, std, seed):
    rng = np.random.default_rng(seed)
    gen = torch.Generator().manual_seed(seed)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    parents = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        if N == 1:
            parents[b] = [-1]
        else:
            parents[b], _ = inputs.make_tree(rng, N, min(8, N - 1), 10, 100)
    S_max = max(P) + 70
    q = (torch.randn(B, N, Hq, d, generator=gen) * std).to(dt)
    k = (torch.randn(B, N, Hkv, d, generator=gen) * std).to(dt)
    v = (torch.randn(B, N, Hkv, d, generator=gen) * std).to(dt)
    cK = (torch.randn(B, Hkv, S_max, d, generator=gen) * std).to(dt)
    cV = (torch.randn(B, Hkv, S_max, d, generator=gen) * std).to(dt)
    return parents, np.array(P, dtype=np.int32), S_max, q, k, v, cK, cV


def run_gpu_attention(dev, parents, P, S_max, q, k, v, cK, cV, base, ws=None):
    B, N, Hq, d = q.shape
    Hkv = k.shape[2]
    dt = q.dtype
    t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    depth = torch.zeros(B, N, dtype=torch.int32, device=dev)
    pos = torch.zeros_like(depth)
    anc = torch.zeros(B, N, dtype=torch.int64, device=dev)
    st = torch.zeros(B, dtype=torch.int32, device=dev)
    Pd = t(P)
    gv.gv_tree_build(t(parents), Pd, depth, pos, anc, st)
    rope = torch.zeros(B, N, d // 2, 2, dtype=torch.float32, device=dev)
    gv.gv_rope_table(pos, d, base, rope)
    shape = gv.attn_shape(B, N, Hq, Hkv, d, S_max, gv.GV_BF16 if dt == torch.bfloat16 else gv.GV_F32)
    if ws is None:
        ws = torch.full((gv.gv_verify_attention_workspace(shape),), 0xFF, dtype=torch.uint8, device=dev)
    tK = torch.zeros(B, Hkv, N, d, dtype=dt, device=dev)
    tV = torch.zeros_like(tK)
    out = torch.zeros(B, N, Hq, d, dtype=dt, device=dev)
    gv.gv_verify_attention(shape, q.to(dev), k.to(dev), v.to(dev), cK.to(dev), cV.to(dev), Pd, rope,
                           anc, tK, tV, out, ws)
    torch.cuda.synchronize()
    return out, tK, tV, pos, anc


@pytest.mark.parametrize("case", range(len(CASES)))
def test_attention_parity(case):
    dev = device()
    dtype, B, N, Hq, Hkv, d, P, base, std = CASES[case]
    parents, P, S_max, q, k, v, cK, cV = _case(dtype, B, N, Hq, Hkv, d, P, base, std, 100 + case)
    out, tK, tV, pos, anc = run_gpu_attention(dev, parents, P, S_max, q, k, v, cK, cV, base)
    depth, rpos, ranc, _ = oracle.tree_build(parents, P)
    np.testing.assert_array_equal(pos.cpu().numpy(), rpos)
    ro, rK, rV = oracle.tree_attention(f64(q), f64(k), f64(v), f64(cK), f64(cV), P, rpos, ranc, base)
    assert np.isfinite(f64(out)).all()
    e = rel_err(f64(out), ro)
    assert e <= TOL_ATTN[dtype], e
    assert rel_err(f64(tK), rK) <= TOL_ROT[dtype]
    np.testing.assert_array_equal(f64(tV), rV)


def test_attention_repeatable_on_reused_workspace():
    """Three calls on one workspace that starts dirty (each on what the
    previous left behind) agree bitwise and with the oracle."""
    dev = device()
    parents, P, S_max, q, k, v, cK, cV = _case("bf16", 2, 60, 32, 8, 128, [700, 1500], 5e5, 1.0, 7)
    shape = gv.attn_shape(2, 60, 32, 8, 128, S_max, gv.GV_BF16)
    ws = torch.full((gv.gv_verify_attention_workspace(shape),), 0xFF, dtype=torch.uint8, device=dev)
    outs = [run_gpu_attention(dev, parents, P, S_max, q, k, v, cK, cV, 5e5, ws)[0] for _ in range(3)]
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])
    ro, _, _ = oracle.tree_attention(f64(q), f64(k), f64(v), f64(cK), f64(cV), P,
                                     oracle.tree_build(parents, P)[1], oracle.tree_build(parents, P)[2], 5e5)
    assert rel_err(f64(outs[2]), ro) <= TOL_ATTN["bf16"]


@pytest.mark.parametrize("case", [4, 6, 9])
def test_rope_apply_matches_the_oracle_and_the_kernel(case):
    # gv_rope_apply over two layers against the oracle's float64 rotation
    # (one bf16 rounding), and the attention with rope = NULL on the rotated
    # inputs against the attention that rotates them itself, bit for bit.
    dtype, B, N, Hq, Hkv, d, P, base, std = CASES[case]
    dev = device()
    parents, P, S_max, q, k, v, cK, cV = _case(dtype, B, N, Hq, Hkv, d, P, base, std, 40 + case)
    out, tK, tV, pos, anc = run_gpu_attention(dev, parents, P, S_max, q, k, v, cK, cV, base)
    rope = torch.zeros(B, N, d // 2, 2, dtype=torch.float32, device=dev)
    gv.gv_rope_table(pos, d, base, rope)
    shape = gv.attn_shape(B, N, Hq, Hkv, d, S_max, gv.GV_BF16)
    q2 = torch.stack([q, q.flip(0) if B > 1 else q]).to(dev)      # two layers
    k2 = torch.stack([k, k]).to(dev)
    q_rot = torch.empty_like(q2)
    k_rot = torch.empty_like(k2)
    gv.gv_rope_apply(shape, q2, k2, rope, q_rot, k_rot)
    torch.cuda.synchronize()
    posn = pos.cpu().numpy()
    for b in range(B):
        ref_q = oracle.rope_rotate(f64(q2[0, b]), posn[b], base)
        ref_k = oracle.rope_rotate(f64(k2[1, b]), posn[b], base)
        assert rel_err(f64(q_rot[0, b]), ref_q) <= TOL_ROT["bf16"]
        assert rel_err(f64(k_rot[1, b]), ref_k) <= TOL_ROT["bf16"]
    # the kernel's own rotation of the tree keys (treeK is [B][Hkv][N][d])
    assert torch.equal(k_rot[0].permute(0, 2, 1, 3), tK)
    tK2 = torch.zeros_like(tK)
    tV2 = torch.zeros_like(tV)
    out2 = torch.zeros_like(out)
    ws = torch.full((gv.gv_verify_attention_workspace(shape),), 0xFF, dtype=torch.uint8, device=dev)
    t32 = torch.as_tensor(P, dtype=torch.int32, device=dev)
    gv.gv_verify_attention(shape, q_rot[0], k_rot[0], v.to(dev), cK.to(dev), cV.to(dev), t32, None, anc, tK2,
                           tV2, out2, ws)
    torch.cuda.synchronize()
    assert torch.equal(out2, out) and torch.equal(tK2, tK) and torch.equal(tV2, tV)
