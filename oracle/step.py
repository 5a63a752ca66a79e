"""Oracle: one whole verify step, composed from the per-stage oracles.

Section 3 of GRIFFIN: draft, then verify all draft tokens in one target
forward pass, then accept.  The composition is:

1. ``tree_build``: depths, positions and ancestor sets from ``parents``;
2. for every layer: ``tree_attention`` (tree scratch K/V for that layer);
3. ``lmhead_logits`` of the final hidden states, then argmax (T = 0) or the
   full logits (T > 0);
4. ``accept_greedy`` or ``accept_sampling``;
5. ``kv_compact`` of the accepted chain into every layer's cache.

``layers`` restricts steps 2 and 5 to the first layers (a bounded sample);
``skip_compact`` leaves out step 5.
"""

import numpy as np

from .tree import tree_build
from .attention import tree_attention
from .lmhead import lmhead_logits, select_argmax
from .accept import accept_greedy, accept_sampling
from .compact import kv_compact


def as_f64(x):
    """Exact widening of a host tensor/array (bf16, fp32, ints) to numpy."""
    if x is None:
        return None
    try:
        import torch
        if isinstance(x, torch.Tensor):
            x = x.detach().cpu()
            if x.is_floating_point():
                return x.double().numpy()
            return x.numpy()
    except ImportError:  # pragma: no cover
        pass
    return np.asarray(x)


def verify_step(inp, layers=None, skip_compact=False):
    """Run the whole step on host copies of ``inp`` (an ``inputs.StepInputs``)."""
    cfg = inp.cfg
    L = cfg["L"] if layers is None else layers
    B, N, D, V = cfg["B"], cfg["N"], cfg["D"], cfg["V"]
    parents = as_f64(inp.parents)
    tokens = as_f64(inp.tokens)
    prefix_len = as_f64(inp.prefix_len)
    depth, pos, anc, status = tree_build(parents, prefix_len)

    attn_out = []
    treeK = []
    treeV = []
    for layer in range(L):
        o, tk, tv = tree_attention(as_f64(inp.q[layer]), as_f64(inp.k_new[layer]),
                                   as_f64(inp.v_new[layer]), as_f64(inp.cacheK[layer]),
                                   as_f64(inp.cacheV[layer]), prefix_len, pos, anc,
                                   cfg["rope_base"])
        attn_out.append(o)
        treeK.append(tk)
        treeV.append(tv)

    logits = lmhead_logits(as_f64(inp.h), as_f64(inp.W))
    T = cfg.get("temperature", 0.0)
    res = dict(depth=depth, pos=pos, anc=anc, tree_status=status, attn_out=attn_out,
               treeK=treeK, treeV=treeV)
    if T == 0.0:
        choice, maxval = select_argmax(logits)
        path, alen, out_tokens, st = accept_greedy(parents, tokens, choice, D, status)
        res.update(choice=choice, maxval=maxval)
    else:
        tl = logits.reshape(B, N, V)
        path, alen, out_tokens, st, margin = accept_sampling(
            parents, tokens, tl, as_f64(inp.draft_logits), as_f64(inp.u_acc),
            as_f64(inp.u_res), D, T, status)
        res.update(logits=logits, margin=margin)
    res.update(path=path, accept_len=alen, out_tokens=out_tokens, seq_status=st)
    if not skip_compact:
        ck, cv, new_len, st2 = kv_compact(np.stack(treeK), np.stack(treeV),
                                          as_f64(inp.cacheK[:L]), as_f64(inp.cacheV[:L]),
                                          path, alen, prefix_len, st)
        res.update(cacheK=ck, cacheV=cv, new_len=new_len, seq_status=st2)
    return res
