"""gv_draft_tree_expand / gv_draft_tree_finish (the dynamic draft tree of a
cycle) through the C ABI against the float64 oracle.  Every output is an
index or a token, compared exactly; the seeds are checked to leave every
score-based decision a margin above 1e-4 in the oracle (fp32 scores on the
GPU, float64 in the oracle: a nearer tie could order either way)."""

import numpy as np
import pytest
import torch

import oracle
from paper_2502_11018_gb300 import gv, inputs
from gpu_util import device

pytestmark = pytest.mark.gpu

MARGIN = 1e-4


def _gpu_tree(cfg, root, steps, ws=None, N=None):
    dev = root.device
    B, k, D, V = cfg["B"], cfg["k"], cfg["D"], cfg["V"]
    N = cfg["N"] if N is None else N
    if ws is None:
        ws = torch.empty(gv.gv_draft_tree_workspace(B, k, D, V), dtype=torch.uint8, device=dev)
    exp_tok, exp_pool = [], []
    for j in range(D):
        et = torch.full((B, k), -7, dtype=torch.int32, device=dev)
        ep = torch.full((B, k), -7, dtype=torch.int32, device=dev)
        gv.gv_draft_tree_expand(j, k, D, steps[j], ws, root_token=root, exp_token=et, exp_pool=ep)
        exp_tok.append(et)
        exp_pool.append(ep)
    parents = torch.full((B, N), -9, dtype=torch.int32, device=dev)
    tokens = torch.full((B, N), -9, dtype=torch.int32, device=dev)
    gv.gv_draft_tree_finish(k, D, V, parents, tokens, ws)
    torch.cuda.synchronize()
    return parents.cpu().numpy(), tokens.cpu().numpy(), [t.cpu().numpy() for t in exp_tok], \
        [p.cpu().numpy() for p in exp_pool]


def _check(cfg, root, steps, N=None):
    B, k, D = cfg["B"], cfg["k"], cfg["D"]
    N = cfg["N"] if N is None else N
    par, tok, etok, epool = _gpu_tree(cfg, root, steps, N=N)
    for b in range(B):
        ref = oracle.draft_tree(int(root[b]), [s[b].float().cpu().numpy() for s in steps], k, D, N)
        assert ref["margin"] > MARGIN, f"seed leaves a near-tie ({ref['margin']:.2e})"
        np.testing.assert_array_equal(par[b], ref["parents"])
        np.testing.assert_array_equal(tok[b], ref["tokens"])
        for j in range(D - 1):
            ids = ref["expanded"][j + 1]
            np.testing.assert_array_equal(epool[j][b], ids)
            np.testing.assert_array_equal(etok[j][b], [ref["pool"]["token"][i] for i in ids])


@pytest.mark.parametrize("name,over", [
    ("draft_small", {}),
    ("draft_small", dict(k=1, D=5, N=6)),          # the greedy chain
    ("draft_small", dict(k=16, D=2, N=64, V=300)),
    ("draft_small", dict(D=1, N=5)),               # the root's top-k only
    ("draft_llama3_8b", {}),
    ("draft_llama2_7b_b4", {}),
    ("draft_small", dict(B=3, k=16, D=16, N=64, V=5000)),   # the largest pool (3857 nodes)
])
def test_draft_tree_parity(name, over):
    cfg = dict(inputs.DRAFT_CONFIGS[name], **over)
    root, steps = inputs.make_draft_logits(cfg, 5, device=device())
    _check(cfg, root, steps)


def test_draft_tree_root_only_and_dirty_workspace():
    cfg = dict(inputs.DRAFT_CONFIGS["draft_small"])
    dev = device()
    root, steps = inputs.make_draft_logits(cfg, 6, device=dev)
    B, k, D, V = cfg["B"], cfg["k"], cfg["D"], cfg["V"]
    ws = torch.full((gv.gv_draft_tree_workspace(B, k, D, V),), 0xFF, dtype=torch.uint8, device=dev)
    par, tok, _, _ = _gpu_tree(cfg, root, steps, ws=ws, N=1)
    assert (par[:, 0] == -1).all() and (tok[:, 0] == root.cpu().numpy()).all()
    # a second tree in the same workspace
    root2, steps2 = inputs.make_draft_logits(cfg, 7, device=dev)
    par2, tok2, _, _ = _gpu_tree(cfg, root2, steps2, ws=ws)
    for b in range(B):
        ref = oracle.draft_tree(int(root2[b]), [s[b].cpu().numpy() for s in steps2], k, D, cfg["N"])
        assert ref["margin"] > MARGIN
        np.testing.assert_array_equal(par2[b], ref["parents"])
        np.testing.assert_array_equal(tok2[b], ref["tokens"])


def test_draft_tree_graph_replay():
    cfg = dict(inputs.DRAFT_CONFIGS["draft_llama2_7b_b4"])
    dev = device()
    root, steps = inputs.make_draft_logits(cfg, 8, device=dev)
    B, k, D, V, N = cfg["B"], cfg["k"], cfg["D"], cfg["V"], cfg["N"]
    ws = torch.empty(gv.gv_draft_tree_workspace(B, k, D, V), dtype=torch.uint8, device=dev)
    parents = torch.zeros((B, N), dtype=torch.int32, device=dev)
    tokens = torch.zeros((B, N), dtype=torch.int32, device=dev)

    def build(stream):
        for j in range(D):
            gv.gv_draft_tree_expand(j, k, D, steps[j], ws, root_token=root, stream=stream)
        gv.gv_draft_tree_finish(k, D, V, parents, tokens, ws, stream=stream)

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        build(s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    eager = (parents.clone(), tokens.clone())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        build(torch.cuda.current_stream())
    parents.zero_()
    tokens.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(parents, eager[0]) and torch.equal(tokens, eager[1])
