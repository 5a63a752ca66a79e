"""GPU parity of the integer steps: tree build, greedy and sampling
acceptance, KV compaction.  Bit-exact against the oracle (sampling decisions:
exact where the oracle's margins exceed the tolerance, otherwise checked to
be a valid outcome of the rule)."""

import numpy as np
import pytest
import torch

import oracle
from oracle.accept import check_sampling_trail
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device, f64

pytestmark = pytest.mark.gpu


def _trees(rng, B, N, D, branch=10, V=1000):
    parents = np.zeros((B, N), dtype=np.int32)
    tokens = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        if N == 1:
            parents[b] = [-1]
            tokens[b] = [int(rng.integers(V))]
        else:
            parents[b], tokens[b] = inputs.make_tree(rng, N, min(D, N - 1), branch, V)
    return parents, tokens


def _tree_gpu(parents, P, dev):
    B, N = parents.shape
    t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    depth = torch.zeros(B, N, dtype=torch.int32, device=dev)
    pos = torch.zeros_like(depth)
    anc = torch.zeros(B, N, dtype=torch.int64, device=dev)
    st = torch.full((B,), 7, dtype=torch.int32, device=dev)
    gv.gv_tree_build(t(parents), t(P), depth, pos, anc, st)
    torch.cuda.synchronize()
    return depth, pos, anc, st


@pytest.mark.parametrize("N", [1, 2, 16, 17, 60, 63, 64])
def test_tree_build_parity(N):
    dev = device()
    rng = np.random.default_rng(N)
    B = 6
    parents, _ = _trees(rng, B, N, 8)
    if N >= 3:
        parents[1, 2] = 2            # self reference
        parents[3, 0] = 0            # root without -1
        parents[4, N - 1] = N        # forward reference
    P = rng.integers(0, 20000, size=B).astype(np.int32)
    depth, pos, anc, st = _tree_gpu(parents, P, dev)
    rd, rp, ra, rs = oracle.tree_build(parents, P)
    np.testing.assert_array_equal(depth.cpu().numpy(), rd)
    np.testing.assert_array_equal(pos.cpu().numpy(), rp)
    np.testing.assert_array_equal(anc.cpu().numpy().view(np.uint64), ra)
    np.testing.assert_array_equal(st.cpu().numpy(), rs)


@pytest.mark.parametrize("seed,N,D", [(0, 60, 6), (1, 60, 8), (2, 16, 4), (3, 64, 10), (4, 1, 0),
                                      (5, 2, 1)])
def test_accept_greedy_parity(seed, N, D):
    dev = device()
    rng = np.random.default_rng(seed)
    B, V = 8, 1000
    parents, tokens = _trees(rng, B, N, D, V=V)
    choice = np.stack([inputs.plant_choices(rng, parents[b], tokens[b], V, p_match=0.6)
                       for b in range(B)])
    if N >= 3:
        # duplicate sibling tokens (legal; resolved by the tie rule)
        kids = inputs.children_of(parents[1])
        if len(kids[0]) >= 2:
            tokens[1, kids[0][1]] = tokens[1, kids[0][0]]
    P = np.full(B, 100, dtype=np.int32)
    depth, pos, anc, st = _tree_gpu(parents, P, dev)
    st_in = np.zeros(B, dtype=np.int32)
    st_in[5] = -2
    st_in_t = torch.as_tensor(st_in, device=dev)
    t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    path = torch.full((B, D + 1), 99, dtype=torch.int32, device=dev)
    alen = torch.full((B,), 99, dtype=torch.int32, device=dev)
    out = torch.full((B, D + 1), 99, dtype=torch.int32, device=dev)
    gv.gv_accept(D, 0.0, t(tokens), anc, depth, t(choice.reshape(-1)), None, None, None, None,
                 path, alen, out, st_in_t)
    torch.cuda.synchronize()
    rp, ra, ro, rs = oracle.accept_greedy(parents, tokens, choice.reshape(-1), D, st_in)
    np.testing.assert_array_equal(path.cpu().numpy(), rp)
    np.testing.assert_array_equal(alen.cpu().numpy(), ra)
    np.testing.assert_array_equal(out.cpu().numpy(), ro)
    np.testing.assert_array_equal(st_in_t.cpu().numpy(), rs)


def test_accept_greedy_depth_over_D():
    dev = device()
    parents = np.array([[-1, 0, 1, 2, 3]], dtype=np.int32)
    tokens = np.array([[5, 1, 2, 3, 4]], dtype=np.int32)
    choice = np.array([1, 2, 3, 4, 9], dtype=np.int32)
    depth, pos, anc, st = _tree_gpu(parents, [0], dev)
    t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    path = torch.zeros(1, 4, dtype=torch.int32, device=dev)
    alen = torch.zeros(1, dtype=torch.int32, device=dev)
    out = torch.zeros(1, 4, dtype=torch.int32, device=dev)
    gv.gv_accept(3, 0.0, t(tokens), anc, depth, t(choice), None, None, None, None, path, alen, out, st)
    torch.cuda.synchronize()
    assert st.item() == gv.GV_ERR_INVALID_TREE and alen.item() == 0
    assert (path.cpu() == -1).all() and (out.cpu() == -1).all()


@pytest.mark.parametrize("seed,V,T,with_q", [(0, 1000, 1.0, True), (1, 32000, 1.0, True), (2, 7, 1.0, True),
                                             (3, 1000, 0.7, True), (4, 1000, 1.0, False),
                                             (5, 32000, 0.7, False), (6, 7, 1.3, False)])
def test_accept_sampling_parity(seed, V, T, with_q):
    # with_q False: no draft distribution (q = 1 for drafted tokens).
    dev = device()
    rng = np.random.default_rng(seed)
    gen = torch.Generator().manual_seed(seed)
    B, N, D = 6, 60 if V > 50 else 9, 8 if V > 50 else 3
    parents, tokens = _trees(rng, B, N, D, V=max(V, 20))
    tl = torch.randn(B, N, V, generator=gen) * 2.0
    dl = tl + torch.randn(B, N, V, generator=gen)
    for b in range(B):
        for c in range(1, N):
            qd = torch.softmax(dl[b, parents[b, c]].double(), 0)
            tokens[b, c] = int(torch.multinomial(qd.float(), 1, generator=gen))
    ua = torch.rand(B, N, generator=gen)
    ur = torch.rand(B, N, generator=gen)
    P = np.zeros(B, dtype=np.int32)
    depth, pos, anc, st = _tree_gpu(parents, P, dev)
    t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    path = torch.zeros(B, D + 1, dtype=torch.int32, device=dev)
    alen = torch.zeros(B, dtype=torch.int32, device=dev)
    out = torch.zeros(B, D + 1, dtype=torch.int32, device=dev)
    ws = torch.empty(gv.gv_accept_workspace(B, V, T), dtype=torch.uint8, device=dev)
    gv.gv_accept(D, T, t(tokens), anc, depth, None, tl.to(dev), dl.to(dev) if with_q else None, ua.to(dev),
                 ur.to(dev), path, alen, out, st, ws)
    torch.cuda.synchronize()
    dl64 = f64(dl) if with_q else None
    rp, ra, ro, rs, margin = oracle.accept_sampling(parents, tokens, f64(tl), dl64, f64(ua),
                                                    f64(ur), D, T)
    gp, ga, go = path.cpu().numpy(), alen.cpu().numpy(), out.cpu().numpy()
    assert (st.cpu().numpy() == 0).all()
    exact = 0
    for b in range(B):
        trail = gp[b, :ga[b]].tolist()
        ok, amb = check_sampling_trail(parents[b], tokens[b], f64(tl[b]), None if dl64 is None else dl64[b],
                                       f64(ua[b]), f64(ur[b]), trail, int(go[b, ga[b] - 1]), T, tol=1e-5)
        assert ok, (b, trail)
        assert go[b, :ga[b] - 1].tolist() == [int(tokens[b, j]) for j in trail[1:]]
        if margin[b] > 1e-4:
            assert gp[b].tolist() == rp[b].tolist() and go[b].tolist() == ro[b].tolist()
            exact += 1
    assert exact >= B // 2


def test_kv_compact_parity():
    dev = device()
    rng = np.random.default_rng(3)
    L, B, Hkv, N, d, D = 3, 4, 2, 60, 128, 8
    S = 300
    parents, tokens = _trees(rng, B, N, D)
    choice = np.stack([inputs.plant_choices(rng, parents[b], tokens[b], 1000, 0.8) for b in range(B)])
    rp, ra, _, _ = oracle.accept_greedy(parents, tokens, choice.reshape(-1), D)
    P = np.array([0, 17, 300, 250], dtype=np.int32)       # sequence 2 overflows S_max
    st_in = np.array([0, 0, 0, -2], dtype=np.int32)
    for dt in (torch.bfloat16, torch.float32):
        gen = torch.Generator().manual_seed(4)
        tK = torch.randn(L, B, Hkv, N, d, generator=gen).to(dt)
        tV = torch.randn(L, B, Hkv, N, d, generator=gen).to(dt)
        cK = torch.randn(L, B, Hkv, S, d, generator=gen).to(dt)
        cV = torch.randn(L, B, Hkv, S, d, generator=gen).to(dt)
        gK, gV = cK.to(dev), cV.to(dev)
        t = lambda a: torch.as_tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
        new_len = torch.zeros(B, dtype=torch.int32, device=dev)
        st = t(st_in)
        gv.gv_kv_compact(D, tK.to(dev), tV.to(dev), gK, gV, t(rp), t(ra), t(P), new_len, st)
        torch.cuda.synchronize()
        oK, oV, onl, ost = oracle.kv_compact(f64(tK), f64(tV), f64(cK), f64(cV), rp, ra, P, st_in)
        np.testing.assert_array_equal(f64(gK), oK)
        np.testing.assert_array_equal(f64(gV), oV)
        np.testing.assert_array_equal(new_len.cpu().numpy(), onl)
        np.testing.assert_array_equal(st.cpu().numpy(), ost)
        assert ost[2] == gv.GV_ERR_CAPACITY
