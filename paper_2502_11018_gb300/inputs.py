"""Seeded synthetic inputs for the verify pass (shared by tests, bench, smoke).

This module only *synthesises* inputs: draft trees, draft tokens, planted
hidden states, random weights and caches, uniforms.  It holds none of the
verify pass's arithmetic (no attention, projection, selection or acceptance)
and imports neither the CUDA library nor the oracle.

Workload shapes follow GRIFFIN's evaluation: batch 1 (Section 5), a dynamic
draft tree of 60 tokens and depth 6 built EAGLE-2 style from top-k
expansions (Appendix C), T in {0, 1} (Section 5), LLaMA-2/LLaMA-3/Mixtral
shaped target models (Section 5).  The MT-Bench / HumanEval / GSM8K prompts
the paper decodes are not used: seeded random weights, caches and trees of
the same shapes stand in for them.
"""

import math
from dataclasses import dataclass, field

import numpy as np
import torch

# --------------------------------------------------------------------------
# Workload configurations.  Layer counts are the public model shapes.
# --------------------------------------------------------------------------

CONFIGS = {
    # One attention layer + LM head, fp32, MHA 8 x 64, vocab 4096, prefix 256,
    # 16-node tree of depth 4 with branching <= 4.
    "tiny_f32": dict(dtype="f32", B=1, L=1, H=512, Hq=8, Hkv=8, d=64, V=4096,
                     P=(256,), N=16, D=4, branch=4, rope_base=10000.0,
                     std_w=0.02, std_kv=0.02, temperature=0.0),
    # LLaMA-2-7B shaped: MHA 32 x 128, vocab 32000, prefix 2048, 60 nodes depth 6.
    "llama2_7b": dict(dtype="bf16", B=1, L=32, H=4096, Hq=32, Hkv=32, d=128, V=32000,
                      P=(2048,), N=60, D=6, branch=10, rope_base=10000.0,
                      std_w=0.02, std_kv=1.0, temperature=0.0),
    # LLaMA-3-8B shaped: GQA 32q / 8kv x 128, vocab 128256, prefix 4096, depth 8.
    "llama3_8b": dict(dtype="bf16", B=1, L=32, H=4096, Hq=32, Hkv=8, d=128, V=128256,
                      P=(4096,), N=60, D=8, branch=10, rope_base=500000.0,
                      std_w=0.02, std_kv=1.0, temperature=0.0),
    # LLaMA-2-13B shaped, batch 4 with ragged prefixes.
    "llama2_13b_b4": dict(dtype="bf16", B=4, L=40, H=5120, Hq=40, Hkv=40, d=128, V=32000,
                          P=(1024, 3072, 6144, 8192), N=60, D=6, branch=10,
                          rope_base=10000.0, std_w=0.02, std_kv=1.0, temperature=0.0),
    # Batched chain speculation (the paper's vLLM throughput appendix): LLaMA-3-8B
    # shape, 16 sequences, each a chain of 2 drafts after the root token
    # (N = 3, D = 2), ragged chat-length prefixes, greedy acceptance.
    "llama3_8b_chain_b16": dict(dtype="bf16", B=16, L=32, H=4096, Hq=32, Hkv=8, d=128, V=128256,
                                P=(512, 768, 1024, 1536), N=3, D=2, branch=1,
                                rope_base=500000.0, std_w=0.02, std_kv=1.0, temperature=0.0),
    # Mixtral-8x7B attention shape, long context, temperature-1 acceptance.
    "mixtral_attn": dict(dtype="bf16", B=1, L=32, H=4096, Hq=32, Hkv=8, d=128, V=32000,
                         P=(16384,), N=60, D=8, branch=10, rope_base=1000000.0,
                         std_w=0.02, std_kv=1.0, temperature=1.0),
}


def config(name, **overrides):
    cfg = dict(CONFIGS[name])
    cfg.update(overrides)
    cfg["name"] = name
    cfg["P"] = tuple(cfg["P"])
    if len(cfg["P"]) != cfg["B"]:
        cfg["P"] = tuple(cfg["P"][i % len(cfg["P"])] for i in range(cfg["B"]))
    cfg.setdefault("S_max", max(cfg["P"]) + 64 + 64)
    return cfg


# --------------------------------------------------------------------------
# Draft trees.
# --------------------------------------------------------------------------

def make_tree(rng, N, D, branch, V):
    """EAGLE-2 style dynamic draft tree with ``N`` nodes (root included).

    Every expanded node proposes ``branch`` candidate children with distinct
    tokens and seeded log-probabilities; a candidate's score is its parent's
    score plus its own log-probability.  The best-scoring chain of first
    candidates is kept down to depth ``D`` (so the tree reaches depth ``D``);
    the remaining ``N - 1 - D`` slots take the best-scoring candidates whose
    parent is already kept.  Nodes are then renumbered breadth first (by
    depth, then by parent, then by candidate rank), so ``parents[i] < i`` and
    the first child of a node is its best candidate.

    Returns ``parents`` (int32[N], ``parents[0] = -1``) and ``tokens``
    (int32[N]; ``tokens[0]`` is the root, i.e. the last committed token).
    """
    assert N >= D + 1, "tree must hold a chain of depth D"
    # Candidate table: id -> (parent id, depth, score, rank, token)
    cand = [(-1, 0, 0.0, 0, int(rng.integers(V)))]
    children = {}

    def expand(u):
        if u in children:
            return children[u]
        par, dep, score, _, _ = cand[u]
        g = np.sort(rng.normal(0.0, 2.0, size=branch))[::-1]
        logp = g - (g.max() + math.log(np.exp(g - g.max()).sum() + 1.0))  # strictly < 0
        toks = rng.choice(V, size=branch, replace=False)
        ids = []
        for r in range(branch):
            cand.append((u, dep + 1, score + float(logp[r]), r, int(toks[r])))
            ids.append(len(cand) - 1)
        children[u] = ids
        return ids

    kept = [0]
    keptset = {0}
    u = 0
    for _ in range(D):
        c = expand(u)[0]
        kept.append(c)
        keptset.add(c)
        u = c
    # Expand every node of depth < D that is kept, repeatedly, best first.
    while len(kept) < N:
        for k in list(kept):
            if cand[k][1] < D:
                expand(k)
        best = None
        for cid in range(1, len(cand)):
            if cid in keptset or cand[cid][0] not in keptset:
                continue
            if best is None or cand[cid][2] > cand[best][2]:
                best = cid
        if best is None:
            raise ValueError(f"branch {branch} and depth {D} cannot hold {N} nodes")
        kept.append(best)
        keptset.add(best)
    # Breadth-first renumbering.
    order = sorted(kept, key=lambda cid: (cand[cid][1], _bfs_key(cand, cid)))
    new_id = {cid: i for i, cid in enumerate(order)}
    parents = np.full(N, -1, dtype=np.int32)
    tokens = np.zeros(N, dtype=np.int32)
    for cid in order:
        i = new_id[cid]
        par = cand[cid][0]
        parents[i] = -1 if par == -1 else new_id[par]
        tokens[i] = cand[cid][4]
    return parents, tokens


def _bfs_key(cand, cid):
    key = []
    while cid != -1:
        key.append(cand[cid][3])
        cid = cand[cid][0]
    return tuple(reversed(key))


def children_of(parents):
    ch = [[] for _ in range(len(parents))]
    for i in range(1, len(parents)):
        ch[int(parents[i])].append(i)
    return ch


def plant_choices(rng, parents, tokens, V, p_match=0.5):
    """Planted target choice per node for greedy verification.

    For a node with children, with probability ``p_match`` the planted choice
    is the token of its first child (so that child matches), otherwise a
    token none of its children carries; leaves get a random token.
    """
    ch = children_of(parents)
    out = np.zeros(len(parents), dtype=np.int32)
    for u in range(len(parents)):
        kids = {int(tokens[c]) for c in ch[u]}
        if ch[u] and rng.random() < p_match:
            out[u] = tokens[ch[u][0]]
        else:
            while True:
                t = int(rng.integers(V))
                if t not in kids:
                    break
            out[u] = t
    return out


# --------------------------------------------------------------------------
# Tensors.
# --------------------------------------------------------------------------

def torch_dtype(cfg):
    return torch.bfloat16 if cfg["dtype"] == "bf16" else torch.float32


def randn(gen, shape, std, dtype, device):
    x = torch.randn(shape, generator=gen, dtype=torch.float32, device=device)
    if std != 1.0:
        x.mul_(std)
    return x.to(dtype)


def planted_hidden(gen, W, targets, alpha=1.0, eps_rel=0.05, weights=None):
    """Rows ``h[r] = sum_k a_k W[t_rk] / |W[t_rk]| + eps * n_r``.

    With ``targets`` of shape ``[rows]`` this is ``alpha * W[t] / |W[t]| +
    eps * n`` (``eps = eps_rel * alpha / sqrt(H)``): the planted token's score
    is about ``alpha * |W[t]|`` while every other score is a small random
    projection, so the planted token is the row's maximum by a wide margin.
    With ``targets`` of shape ``[rows][k]`` and per-column ``weights`` the row
    is a weighted mix (used to shape temperature-1 target distributions:
    the score of ``t_rk`` is then about ``weights[k]``).
    """
    Wf = W.float()
    t = torch.as_tensor(targets, device=W.device, dtype=torch.long)
    H = W.shape[1]
    if t.dim() == 1:
        rowsW = Wf[t]
        h = alpha * rowsW / rowsW.norm(dim=1, keepdim=True)
        eps = eps_rel * alpha / math.sqrt(H)
    else:
        wts = torch.as_tensor(weights, device=W.device, dtype=torch.float32)
        h = torch.zeros(t.shape[0], H, device=W.device)
        for k in range(t.shape[1]):
            rowsW = Wf[t[:, k]]
            h += wts[k] * rowsW / (rowsW.norm(dim=1, keepdim=True) ** 2)
        eps = eps_rel / math.sqrt(H)
    n = torch.randn(h.shape, generator=gen, device=W.device, dtype=torch.float32)
    return (h + eps * n).to(W.dtype)


@dataclass
class StepInputs:
    """All inputs of one verify step (device or host tensors)."""
    cfg: dict
    parents: torch.Tensor            # int32 [B][N]
    tokens: torch.Tensor             # int32 [B][N]
    prefix_len: torch.Tensor         # int32 [B]
    planted: torch.Tensor            # int32 [B][N]  planted greedy choice (T = 0)
    q: torch.Tensor                  # [L][B][N][Hq][d]
    k_new: torch.Tensor              # [L][B][N][Hkv][d]
    v_new: torch.Tensor              # [L][B][N][Hkv][d]
    cacheK: torch.Tensor             # [L][B][Hkv][S_max][d]
    cacheV: torch.Tensor             # [L][B][Hkv][S_max][d]
    h: torch.Tensor                  # [B*N][H]
    W: torch.Tensor                  # [V][H]
    draft_logits: torch.Tensor = None  # fp32 [B][N][V]   (T > 0)
    u_acc: torch.Tensor = None         # fp32 [B][N]      (T > 0)
    u_res: torch.Tensor = None         # fp32 [B][N]      (T > 0)
    extra: dict = field(default_factory=dict)


def make_step_inputs(cfg, seed, device="cpu", layers=None):
    """Build one seeded verify step for ``cfg`` on ``device``.

    ``layers`` overrides the layer count (tests use fewer layers than the
    bench; each layer's tensors are drawn independently).
    """
    L = cfg["L"] if layers is None else layers
    B, N, D, V, H = cfg["B"], cfg["N"], cfg["D"], cfg["V"], cfg["H"]
    Hq, Hkv, d, S_max = cfg["Hq"], cfg["Hkv"], cfg["d"], cfg["S_max"]
    dt = torch_dtype(cfg)
    rng = np.random.default_rng(seed)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))

    parents = np.zeros((B, N), dtype=np.int32)
    tokens = np.zeros((B, N), dtype=np.int32)
    planted = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        parents[b], tokens[b] = make_tree(rng, N, D, cfg["branch"], V)
        planted[b] = plant_choices(rng, parents[b], tokens[b], V)

    W = randn(gen, (V, H), cfg["std_w"], dt, device)
    std = cfg["std_kv"]
    q = randn(gen, (L, B, N, Hq, d), std, dt, device)
    k_new = randn(gen, (L, B, N, Hkv, d), std, dt, device)
    v_new = randn(gen, (L, B, N, Hkv, d), std, dt, device)
    cacheK = randn(gen, (L, B, Hkv, S_max, d), std, dt, device)
    cacheV = randn(gen, (L, B, Hkv, S_max, d), std, dt, device)

    draft_logits = u_acc = u_res = None
    T = cfg.get("temperature", 0.0)
    if T > 0.0:
        # Temperature-1 workload: each node's target distribution is shaped by
        # three planted tokens (scores about 10, 9, 8 over a near-flat tail);
        # the draft logits carry the same planted scores plus N(0, 1) noise on
        # every token; each node's children are then drawn i.i.d. from the
        # draft distribution of the parent, as speculative sampling assumes.
        hot = np.stack([rng.choice(V, size=3, replace=False) for _ in range(B * N)])
        h = planted_hidden(gen, W, hot, weights=[10.0, 9.0, 8.0])
        dl = torch.randn((B, N, V), generator=gen, device=device, dtype=torch.float32)
        hot_t = torch.as_tensor(hot, device=device, dtype=torch.long).view(B, N, 3)
        dl.scatter_add_(2, hot_t, torch.tensor([10.0, 9.0, 8.0], device=device).expand(B, N, 3).contiguous())
        draft_logits = dl
        for b in range(B):
            ch = children_of(parents[b])
            for u in range(N):
                if not ch[u]:
                    continue
                qd = torch.softmax(dl[b, u].double() / T, dim=0)
                draws = torch.multinomial(qd.float(), len(ch[u]), replacement=True, generator=gen)
                for c, x in zip(ch[u], draws.tolist()):
                    tokens[b, c] = x
        u_acc = torch.rand((B, N), generator=gen, device=device, dtype=torch.float32)
        u_res = torch.rand((B, N), generator=gen, device=device, dtype=torch.float32)
    else:
        h = planted_hidden(gen, W, planted.reshape(-1))

    def i32(a):
        return torch.as_tensor(a, dtype=torch.int32).to(device)

    return StepInputs(cfg=dict(cfg, L=L), parents=i32(parents), tokens=i32(tokens),
                      prefix_len=i32(np.array(cfg["P"], dtype=np.int32)), planted=i32(planted),
                      q=q, k_new=k_new, v_new=v_new, cacheK=cacheK, cacheV=cacheV,
                      h=h, W=W, draft_logits=draft_logits, u_acc=u_acc, u_res=u_res)


# --------------------------------------------------------------------------
# Token-alignable training pass (Section 4.1): draft logits over training
# sequences, ground-truth tokens, draft / target features and the earlier
# passes' predictable masks.  Shapes follow the paper's training setup for a
# LLaMA-2-7B-sized drafter (vocabulary 32000, hidden 4096, N = 3 passes, top-3
# alignment); ShareGPT itself is not used: seeded random values of the same
# shapes stand in for it.
# --------------------------------------------------------------------------

TAT_CONFIGS = {
    # ragged sizes (no 16-byte multiple rows), every pass
    "tat_small": dict(B=2, T=37, V=1001, H=72, k=3, n=3, logits="f32", feat="bf16"),
    # a training batch of 4 sequences x 2048 tokens, fp32 logits
    "tat_llama2_7b": dict(B=4, T=2048, V=32000, H=4096, k=3, n=3, logits="f32", feat="bf16"),
}


@dataclass
class TatInputs:
    cfg: dict
    logits: torch.Tensor        # [B][T][V]
    tokens: torch.Tensor        # int32 [B][T]
    feat_draft: torch.Tensor    # [B][T][H]
    feat_target: torch.Tensor   # [B][T][H]
    mbar_prev: torch.Tensor     # uint8 [n-1][B][T] (None for n = 1)


def make_tat_inputs(cfg, seed, device="cpu", p_plant=0.7, p_prev=0.7):
    """Seeded inputs of one training pass.  Logits ~ N(0, 1); for a fraction
    ``p_plant`` of the positions the ground-truth token is the one at rank
    0..4 of its row (ranks 3 and 4 fall outside a top-3), else a uniform
    token, so that the predictable mask is mixed; features ~ N(0, 1); the
    earlier passes' masks are Bernoulli(``p_prev``)."""
    B, T, V, H, n = cfg["B"], cfg["T"], cfg["V"], cfg["H"], cfg["n"]
    ldt = torch.bfloat16 if cfg["logits"] == "bf16" else torch.float32
    fdt = torch.bfloat16 if cfg["feat"] == "bf16" else torch.float32
    gen = torch.Generator(device="cpu")
    gen.manual_seed(int(seed))
    rng = np.random.default_rng(seed)
    logits = torch.randn((B * T, V), generator=gen, dtype=torch.float32).to(ldt)
    tokens = rng.integers(0, V, size=B * T)
    plant = rng.random(B * T) < p_plant
    ranks = rng.integers(0, 5, size=B * T)
    top = torch.topk(logits.float(), k=min(5, V), dim=1).indices.numpy()
    for r in np.nonzero(plant)[0]:
        tokens[r] = top[r, min(ranks[r], top.shape[1] - 1)]
    fd = torch.randn((B, T, H), generator=gen, dtype=torch.float32).to(fdt)
    ft = torch.randn((B, T, H), generator=gen, dtype=torch.float32).to(fdt)
    prev = None
    if n > 1:
        prev = torch.from_numpy((rng.random((n - 1, B, T)) < p_prev).astype(np.uint8))
    return TatInputs(cfg=dict(cfg), logits=logits.view(B, T, V).to(device),
                     tokens=torch.from_numpy(tokens.astype(np.int32)).view(B, T).to(device),
                     feat_draft=fd.to(device), feat_target=ft.to(device),
                     mbar_prev=None if prev is None else prev.to(device))



# --------------------------------------------------------------------------
# Target decoder-layer weights for the whole verify forward (LLaMA-style:
# RMSNorm, Q/K/V/O projections, SwiGLU MLP).  FFN widths are the public model
# shapes; weights ~ N(0, 0.02), norm weights ~ 1 + N(0, 0.05), the draft
# tokens' input embeddings ~ N(0, 1).
# --------------------------------------------------------------------------

FFN = {"llama2_7b": 11008, "llama3_8b": 14336, "llama2_13b_b4": 13824, "llama3_8b_chain_b16": 14336}


@dataclass
class ForwardWeights:
    F: int
    h0: torch.Tensor          # [B*N][H]  embeddings of the tree's tokens
    attn_norm: torch.Tensor   # [L][H]
    Wqkv: torch.Tensor        # [L][(Hq + 2 Hkv) * d][H]: Wq rows, then Wk, then Wv
    Wo: torch.Tensor          # [L][H][Hq*d]
    mlp_norm: torch.Tensor    # [L][H]
    Wgu: torch.Tensor         # [L][2F][H]  gate rows, then up rows
    Wd: torch.Tensor          # [L][H][F]
    final_norm: torch.Tensor  # [H]


def make_forward_weights(cfg, seed, device="cpu", layers=None, F=None):
    L = cfg["L"] if layers is None else layers
    F = FFN[cfg["name"]] if F is None else F
    B, N, H, Hq, Hkv, d = cfg["B"], cfg["N"], cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["d"]
    dt = torch.bfloat16
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) + 77)
    std = cfg["std_w"]

    def norm_w(*shape):
        return (1.0 + 0.05 * torch.randn(shape, generator=gen, device=device, dtype=torch.float32)).to(dt)

    return ForwardWeights(
        F=F, h0=randn(gen, (B * N, H), 1.0, dt, device),
        attn_norm=norm_w(L, H), Wqkv=randn(gen, (L, (Hq + 2 * Hkv) * d, H), std, dt, device),
        Wo=randn(gen, (L, H, Hq * d), std, dt, device), mlp_norm=norm_w(L, H),
        Wgu=randn(gen, (L, 2 * F, H), std, dt, device), Wd=randn(gen, (L, H, F), std, dt, device),
        final_norm=norm_w(H))


# --------------------------------------------------------------------------
# Token-Guided Fusion (Section 4.2, Eqs. 6-8) of the draft model.  Rows are
# the positions the draft model reads in one call (the 60 nodes of a
# verified tree); d is the target's hidden size and e the expansion width
# (11008 for the LLaMA-2-7B drafter of the Implementation Details appendix).
# Features F ~ N(0, 1) (the target's hidden states), token embeddings
# x ~ N(0, 0.02) (the scale of a LLaMA embedding table), projection weights
# ~ N(0, 0.02), biases ~ N(0, 0.02), layer-norm gains ~ 1 + N(0, 0.05).
# --------------------------------------------------------------------------

TGF_CONFIGS = {
    "tgf_small": dict(rows=7, d=128, e=520),           # ragged expansion (partial tiles)
    "tgf_llama2_7b": dict(rows=60, d=4096, e=11008),
    "tgf_llama2_7b_r256": dict(rows=256, d=4096, e=11008),
}

TGF_WEIGHTS = ("Wm", "bm", "g_h", "b_h", "g_x", "b_x", "Wu", "bu", "Wd", "bd")


@dataclass
class TgfInputs:
    cfg: dict
    F: torch.Tensor      # [rows][d]
    x: torch.Tensor      # [rows][d]
    w: dict              # TGF_WEIGHTS -> bf16 tensors (Wm [d][2d], Wu [e][2d], Wd [d][e], vectors)


def make_tgf_inputs(cfg, seed, device="cpu"):
    rows, d, e = cfg["rows"], cfg["d"], cfg["e"]
    dt = torch.bfloat16
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) + 313)

    def gain(n):
        return (1.0 + 0.05 * torch.randn((n,), generator=gen, device=device, dtype=torch.float32)).to(dt)

    w = {"Wm": randn(gen, (d, 2 * d), 0.02, dt, device), "bm": randn(gen, (d,), 0.02, dt, device),
         "g_h": gain(d), "b_h": randn(gen, (d,), 0.02, dt, device),
         "g_x": gain(d), "b_x": randn(gen, (d,), 0.02, dt, device),
         "Wu": randn(gen, (e, 2 * d), 0.02, dt, device), "bu": randn(gen, (e,), 0.02, dt, device),
         "Wd": randn(gen, (d, e), 0.02, dt, device), "bd": randn(gen, (d,), 0.02, dt, device)}
    return TgfInputs(cfg=dict(cfg), F=randn(gen, (rows, d), 1.0, dt, device),
                     x=randn(gen, (rows, d), 0.02, dt, device), w=w)


# --------------------------------------------------------------------------
# Dynamic draft trees (top-k expansion steps + rerank).  One cycle of a
# LLaMA-3-8B drafter: k = 10 tokens per expanded node, D = 6 steps, N = 60
# tree nodes; the logits of each step are synthetic stand-ins for the draft
# model's: N(0, 1) over the vocabulary plus eight planted tokens per row
# raised by 14, 12, 11, 10, 9, 8, 7, 6 (a peaked distribution, top-1
# probability about 0.7, like a trained drafter's).
# --------------------------------------------------------------------------

DRAFT_CONFIGS = {
    "draft_small": dict(B=2, k=4, D=3, N=12, V=1000, dtype="f32"),
    "draft_llama3_8b": dict(B=1, k=10, D=6, N=60, V=128256, dtype="f32"),
    "draft_llama2_7b_b4": dict(B=4, k=10, D=6, N=60, V=32000, dtype="bf16"),
}

DRAFT_BOOSTS = (14.0, 12.0, 11.0, 10.0, 9.0, 8.0, 7.0, 6.0)


def make_draft_logits(cfg, seed, device="cpu"):
    """(root_token int32 [B], [step 0 logits [B][1][V], step j logits [B][k][V] ...])."""
    B, k, D, V = cfg["B"], cfg["k"], cfg["D"], cfg["V"]
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) + 919)
    dt = torch.bfloat16 if cfg["dtype"] == "bf16" else torch.float32
    steps = []
    boosts = torch.tensor(DRAFT_BOOSTS, dtype=torch.float32, device=device)
    for j in range(D):
        rows = 1 if j == 0 else k
        x = torch.randn((B, rows, V), generator=gen, dtype=torch.float32, device=device)
        nb = min(len(DRAFT_BOOSTS), V)
        pick = torch.rand((B, rows, V), generator=gen, device=device).argsort(dim=2)[:, :, :nb]
        x.scatter_add_(2, pick, boosts[:nb].expand(B, rows, nb).contiguous())
        steps.append(x.to(dt))
    root = torch.randint(0, V, (B,), generator=gen, dtype=torch.int32, device=device)
    return root, steps
