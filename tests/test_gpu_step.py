"""Whole verify step through the C ABI (VerifyStep) against the composed
float64 oracle, on every workload shape with a reduced layer count.

Checked per step: tree outputs bit-exact; every layer's attention output and
rotated tree keys within tolerance, tree values exact; argmax choices
bit-exact (planted); accepted path, length and emitted tokens bit-exact for
greedy acceptance; for temperature-1 acceptance, the GPU's trail must be a
valid outcome of the rule under the oracle's float64 probabilities and equal
the oracle's trail wherever the oracle's margins exceed 1e-4; the compacted
caches hold the GPU's tree rows at the accepted slots and the original bytes
everywhere else."""

import numpy as np
import pytest
import torch

import oracle
from oracle.accept import check_sampling_trail
from paper_2502_11018_gb300 import inputs
from paper_2502_11018_gb300.step import VerifyStep
from gpu_util import device, f64, rel_err, to_device, TOL_ATTN, TOL_ROT

pytestmark = pytest.mark.gpu

STEPS = [("tiny_f32", 1, 1), ("tiny_f32", 1, 2), ("llama2_7b", 1, 3), ("llama3_8b", 2, 4),
         ("llama2_13b_b4", 1, 5), ("mixtral_attn", 1, 6), ("llama3_8b_chain_b16", 1, 7)]


def check_step(inp, step, ref, graph=False):
    cfg = inp.cfg
    kind = cfg["dtype"]
    B, N, D = cfg["B"], cfg["N"], cfg["D"]
    np.testing.assert_array_equal(step.depth.cpu().numpy(), ref["depth"])
    np.testing.assert_array_equal(step.pos.cpu().numpy(), ref["pos"])
    np.testing.assert_array_equal(step.anc.cpu().numpy().view(np.uint64), ref["anc"])
    for layer in range(cfg["L"]):
        assert rel_err(f64(step.attn_out[layer]), ref["attn_out"][layer]) <= TOL_ATTN[kind]
        assert rel_err(f64(step.treeK[layer]), ref["treeK"][layer]) <= TOL_ROT[kind]
        np.testing.assert_array_equal(f64(step.treeV[layer]), ref["treeV"][layer])
    path = step.path.cpu().numpy()
    alen = step.accept_len.cpu().numpy()
    out = step.out_tokens.cpu().numpy()
    if cfg.get("temperature", 0.0) == 0.0:
        np.testing.assert_array_equal(step.ids.cpu().numpy(), ref["choice"])
        np.testing.assert_array_equal(step.ids.cpu().numpy(), inp.planted.numpy().reshape(-1))
        np.testing.assert_array_equal(path, ref["path"])
        np.testing.assert_array_equal(alen, ref["accept_len"])
        np.testing.assert_array_equal(out, ref["out_tokens"])
    else:
        tl = ref["logits"].reshape(B, N, -1)
        parents = inp.parents.numpy()
        tokens = inp.tokens.numpy()
        for b in range(B):
            trail = path[b, :alen[b]].tolist()
            ok, _ = check_sampling_trail(parents[b], tokens[b], tl[b], f64(inp.draft_logits[b]),
                                         f64(inp.u_acc[b]), f64(inp.u_res[b]), trail,
                                         int(out[b, alen[b] - 1]), cfg["temperature"], tol=1e-4)
            assert ok, trail
            if ref["margin"][b] > 1e-4:
                assert path[b].tolist() == ref["path"][b].tolist()
                assert out[b].tolist() == ref["out_tokens"][b].tolist()
    assert (step.seq_status.cpu().numpy() == 0).all()
    P = inp.prefix_len.numpy()
    np.testing.assert_array_equal(step.new_len.cpu().numpy(), P + alen)
    gK = step.inp.cacheK.cpu()
    tK = step.treeK.cpu()
    for b in range(B):
        lo, hi = int(P[b]), int(P[b] + alen[b])
        for t in range(alen[b]):
            assert torch.equal(gK[:cfg["L"], b, :, lo + t], tK[:, b, :, path[b, t]])
        assert torch.equal(gK[:cfg["L"], b, :, :lo], inp.cacheK[:cfg["L"], b, :, :lo])
        assert torch.equal(gK[:cfg["L"], b, :, hi:], inp.cacheK[:cfg["L"], b, :, hi:])


@pytest.mark.parametrize("name,layers,seed", STEPS)
def test_step_parity(name, layers, seed):
    dev = device()
    cfg = inputs.config(name)
    inp = inputs.make_step_inputs(cfg, seed, device="cpu", layers=layers)
    step = VerifyStep(to_device(inp, dev))
    step.run()
    torch.cuda.synchronize()
    ref = oracle.verify_step(inp, skip_compact=True)
    check_step(inp, step, ref)


def test_step_graph_replay_matches_eager():
    dev = device()
    cfg = inputs.config("llama3_8b")
    inp = inputs.make_step_inputs(cfg, 9, device="cpu", layers=2)
    step = VerifyStep(to_device(inp, dev))
    step.run()
    torch.cuda.synchronize()
    eager = (step.attn_out.clone(), step.ids.clone(), step.path.clone(), step.out_tokens.clone())
    step.capture()
    for _ in range(3):
        step.replay()
    torch.cuda.synchronize()
    assert torch.equal(step.attn_out, eager[0])
    assert torch.equal(step.ids, eager[1])
    assert torch.equal(step.path, eager[2])
    assert torch.equal(step.out_tokens, eager[3])


@pytest.mark.parametrize("name,layers", [("llama3_8b", 5), ("mixtral_attn", 3)])
def test_step_from_host_matches_device(name, layers):
    """The host-fed graph (per-layer inputs copied on a side stream while the
    earlier layers run) gives the same bits as the step on device inputs;
    the device inputs are overwritten after capture, so the replay must copy
    them."""
    dev = device()
    cfg = inputs.config(name)
    inp = inputs.make_step_inputs(cfg, 11, device="cpu", layers=layers)
    ref = VerifyStep(to_device(inp, dev))
    # the reference issues the attention in the host-fed step's layer groups
    # (one multi-layer call per group cuts the work the same way)
    ready = {}
    for a, _ in ref._copy_groups(layers):
        ready[a] = torch.cuda.Event()
        ready[a].record()
    ref.tree()
    ref.attention_layers(ready=ready)
    ref.lmhead()
    ref.accept()
    ref.compact()
    ref.join_merges()
    torch.cuda.synchronize()
    step = VerifyStep(to_device(inp, dev))
    host, res = step.host_buffers()
    g = step.capture_from_host(host, res)
    for n in ("q", "k_new", "v_new", "h"):
        getattr(step.inp, n).zero_()
    step.inp.tokens.fill_(-1)
    res.fill_(-7)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(step.attn_out, ref.attn_out)
    assert torch.equal(step.treeK, ref.treeK) and torch.equal(step.treeV, ref.treeV)
    if ref.ids is not None:
        assert torch.equal(step.ids, ref.ids)
    else:
        assert torch.equal(step.logits, ref.logits)
    B, D = cfg["B"], cfg["D"]
    assert torch.equal(res[:B], ref.accept_len.cpu())
    assert torch.equal(res[B:B + B * (D + 1)].view(B, D + 1), ref.out_tokens.cpu())
    assert torch.equal(res[B + B * (D + 1):].view(B, D + 1), ref.path.cpu())


@pytest.mark.parametrize("name,layers", [("llama3_8b", 7), ("tiny_f32", 4), ("llama3_8b_chain_b16", 4)])
def test_side_merges_match_sequential_layers(name, layers):
    # The per-layer schedule (splits in layer order, each merge on a second
    # stream, workspaces in rotation) gives the outputs of calling
    # gv_verify_attention layer by layer, bit for bit, eagerly and replayed.
    dev = device()
    cfg = inputs.config(name)
    inp = inputs.make_step_inputs(cfg, 13, device="cpu", layers=layers)
    step = VerifyStep(to_device(inp, dev), layers_call=False)
    step.tree()
    for layer in range(layers):
        step.attention(layer)
    torch.cuda.synchronize()
    seq = (step.attn_out.clone(), step.treeK.clone(), step.treeV.clone())
    step.attn_out.zero_()
    for ws in step.attn_ws_slots:
        ws.fill_(0xFF)
    step.attention_layers()
    step.join_merges()
    torch.cuda.synchronize()
    assert torch.equal(step.attn_out, seq[0])
    assert torch.equal(step.treeK, seq[1]) and torch.equal(step.treeV, seq[2])
    step.attn_out.zero_()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        cur = torch.cuda.current_stream()
        step.attention_layers(cur)
        step.join_merges(cur)
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(step.attn_out, seq[0])


@pytest.mark.parametrize("name,layers", [("llama3_8b", 6), ("llama3_8b_chain_b16", 3), ("llama2_7b", 2)])
def test_layers_call_matches_per_layer_schedule(name, layers):
    # One gv_verify_attention_layers call for every layer against the
    # per-layer schedule: the tree K/V scratch bit for bit, the outputs within
    # the attention tolerance (the two cut the keys differently), eagerly and
    # replayed from a CUDA graph (the replays repeat the eager bits).
    dev = device()
    cfg = inputs.config(name)
    inp = inputs.make_step_inputs(cfg, 17, device="cpu", layers=layers)
    d_inp = to_device(inp, dev)
    per = VerifyStep(d_inp, layers_call=False)
    per.tree()
    per.attention_layers()
    per.join_merges()
    step = VerifyStep(d_inp)
    assert step.layers_call
    step.tree()
    step.attention_layers()
    torch.cuda.synchronize()
    assert torch.equal(step.treeK, per.treeK) and torch.equal(step.treeV, per.treeV)
    for layer in range(layers):
        assert rel_err(f64(step.attn_out[layer]), f64(per.attn_out[layer])) <= TOL_ATTN["bf16"]
    eager = step.attn_out.clone()
    step.attn_out.zero_()
    step.attn_ws_layers.fill_(0xFF)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step.attention_layers(torch.cuda.current_stream())
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(step.attn_out, eager)
