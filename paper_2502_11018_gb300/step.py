"""One whole verify step through the C ABI, with torch-allocated buffers.

``VerifyStep`` owns the outputs and workspaces of one workload and issues the
five calls of include/gv.h in order on one stream (GRIFFIN Section 3: draft,
then one verify forward over every draft token, then accept):

1. ``gv_tree_build`` and ``gv_rope_table`` (RoPE cos/sin shared by all layers);
2. the attention of every layer.  A layer's queries, keys and values are
   inputs of the step, so the layers are independent problems: on the bf16
   path (G * N <= 256) one ``gv_verify_attention_layers`` call runs all of
   them in one persistent launch; otherwise ``gv_verify_attention_split`` for
   every layer (per-layer tree K/V scratch), each layer's
   ``gv_verify_attention_merge`` on a second stream beside the next layers'
   splits (a workspace per layer);
3. ``gv_lmhead_select`` (argmax for T = 0, fp32 logits + LSE for T > 0);
4. ``gv_accept``;
5. ``gv_kv_compact`` into every layer's cache.

No host synchronisation happens inside ``run``; it can be captured into a
CUDA graph (``capture``/``replay``).
"""

import math

import torch

from . import gv
from .inputs import StepInputs


class VerifyStep:
    # Attention workspaces in rotation (a layer's merge may still read one):
    # None gives every layer its own, so no split waits for an earlier merge.
    # A wait on a merge in the split stream measured slower than the merges
    # save (13.3 against 12.8 us a layer with 3 workspaces; 11.0 with one
    # per layer, LLaMA-3-8B shape).
    ATTN_SLOTS = None

    def __init__(self, inp: StepInputs, layers_call=None):
        """``layers_call``: run every layer's attention in one
        gv_verify_attention_layers call (None: whenever the shape allows it;
        False: the per-layer split/merge calls)."""
        cfg = inp.cfg
        self.inp = inp
        self.cfg = cfg
        dev = inp.q.device
        if dev.type != "cuda":
            raise ValueError("VerifyStep needs device tensors")
        L, B, N, D, V, H = cfg["L"], cfg["B"], cfg["N"], cfg["D"], cfg["V"], cfg["H"]
        Hq, Hkv, d, S_max = cfg["Hq"], cfg["Hkv"], cfg["d"], cfg["S_max"]
        dt = inp.q.dtype
        self.dt_code = gv.dtype_code(inp.q)
        self.T = float(cfg.get("temperature", 0.0))
        i32 = dict(dtype=torch.int32, device=dev)
        self.depth = torch.zeros(B, N, **i32)
        self.pos = torch.zeros(B, N, **i32)
        self.anc = torch.zeros(B, N, dtype=torch.int64, device=dev)
        self.seq_status = torch.zeros(B, **i32)
        self.rope = torch.zeros(B, N, d // 2, 2, dtype=torch.float32, device=dev)
        self.treeK = torch.zeros(L, B, Hkv, N, d, dtype=dt, device=dev)
        self.treeV = torch.zeros(L, B, Hkv, N, d, dtype=dt, device=dev)
        self.attn_out = torch.zeros(L, B, N, Hq, d, dtype=dt, device=dev)
        self.shape = gv.attn_shape(B, N, Hq, Hkv, d, S_max, self.dt_code)
        ws = gv.gv_verify_attention_workspace(self.shape)
        slots = L if self.ATTN_SLOTS is None else min(L, self.ATTN_SLOTS)
        self.attn_ws_slots = [torch.empty(max(ws, 256), dtype=torch.uint8, device=dev) for _ in range(slots)]
        self.attn_ws = self.attn_ws_slots[0]
        self.merge_stream = torch.cuda.Stream(device=dev)
        # bf16 with G * N <= 256: every layer's attention in one call
        self.layers_call = gv.gv_verify_attention_layers_workspace(self.shape, L) > 0 and layers_call is not False
        if self.layers_call:
            self.attn_ws_layers = torch.empty(gv.gv_verify_attention_layers_workspace(self.shape, L),
                                              dtype=torch.uint8, device=dev)
        # bf16 (d = 128): every layer's queries and tree keys are rotated by
        # one gv_rope_apply ahead of the splits, which then take rope = NULL
        self.prerotate = not self.layers_call and self.dt_code == gv.GV_BF16 and d == 128
        if self.prerotate:
            self.q_rot = torch.empty(L, B, N, Hq, d, dtype=dt, device=dev)
            self.k_rot = torch.empty(L, B, N, Hkv, d, dtype=dt, device=dev)
        self._split_ev = [torch.cuda.Event() for _ in range(L)]
        self._merge_ev = [torch.cuda.Event() for _ in range(L)]
        rows = B * N
        if self.T == 0.0:
            self.lm_mode = gv.GV_SELECT_ARGMAX
            self.ids = torch.zeros(rows, **i32)
            self.vals = torch.zeros(rows, dtype=torch.float32, device=dev)
            self.logits = self.row_max = self.row_lse = None
        else:
            self.lm_mode = gv.GV_SELECT_LOGITS
            self.ids = self.vals = None
            self.logits = torch.zeros(rows, V, dtype=torch.float32, device=dev)
            self.row_max = torch.zeros(rows, dtype=torch.float32, device=dev)
            self.row_lse = torch.zeros(rows, dtype=torch.float32, device=dev)
        lw = gv.gv_lmhead_workspace(rows, H, V, self.dt_code, self.lm_mode, 1)
        self.lm_ws = torch.empty(max(lw, 256), dtype=torch.uint8, device=dev)
        # The step's result (accept_len, out_tokens, path) in one buffer, so
        # that a host-fed step reads it back with one copy.
        self.result = torch.zeros(B + 2 * B * (D + 1), **i32)
        self.accept_len = self.result[:B]
        self.out_tokens = self.result[B:B + B * (D + 1)].view(B, D + 1)
        self.path = self.result[B + B * (D + 1):].view(B, D + 1)
        aw = gv.gv_accept_workspace(B, V, self.T)
        self.acc_ws = torch.empty(max(aw, 256), dtype=torch.uint8, device=dev)
        self.new_len = torch.zeros(B, **i32)
        self.graph = None

    # -------------------------------------------------------------- stages --
    def tree(self, stream=None):
        i = self.inp
        gv.gv_tree_build(i.parents, i.prefix_len, self.depth, self.pos, self.anc, self.seq_status,
                         stream)
        gv.gv_rope_table(self.pos, self.cfg["d"], self.cfg["rope_base"], self.rope, stream)

    def attention(self, layer, stream=None):
        """One layer, both halves on ``stream`` (its merged output ready after it)."""
        i = self.inp
        gv.gv_verify_attention(self.shape, i.q[layer], i.k_new[layer], i.v_new[layer],
                               i.cacheK[layer], i.cacheV[layer], i.prefix_len, self.rope, self.anc,
                               self.treeK[layer], self.treeV[layer], self.attn_out[layer],
                               self.attn_ws, stream)

    def attention_layers(self, stream=None, ready=None):
        """Every layer's attention: one ``gv_verify_attention_layers`` call
        (one per group of layers when ``ready`` is given); else the splits on
        ``stream`` in layer order, each layer's merge on ``merge_stream`` after
        its split.  ``ready`` maps a layer to an event that the layers from it
        on wait for (their inputs' copy).  The caller joins the merges with
        ``join_merges`` before it needs the outputs (or ends a graph
        capture)."""
        i = self.inp
        L = self.cfg["L"]
        cur = stream if stream is not None else torch.cuda.current_stream()
        if self.layers_call:
            # one call per group of layers whose inputs arrive together
            starts = sorted(ready) if ready is not None else [0]
            for a, b in zip(starts, starts[1:] + [L]):
                if ready is not None:
                    cur.wait_event(ready[a])
                gv.gv_verify_attention_layers(self.shape, i.q[a:b], i.k_new[a:b], i.v_new[a:b], i.cacheK[a:b],
                                              i.cacheV[a:b], i.prefix_len, self.rope, self.anc, self.treeK[a:b],
                                              self.treeV[a:b], self.attn_out[a:b], self.attn_ws_layers, cur)
            return
        side = self.merge_stream
        side.wait_stream(cur)
        n = len(self.attn_ws_slots)
        starts = sorted(ready) if ready is not None else [0]
        ends = {a: b for a, b in zip(starts, starts[1:] + [L])}
        for layer in range(L):
            if ready is not None and layer in ready:
                cur.wait_event(ready[layer])
            if self.prerotate and layer in ends:
                e = ends[layer]
                gv.gv_rope_apply(self.shape, i.q[layer:e], i.k_new[layer:e], self.rope, self.q_rot[layer:e],
                                 self.k_rot[layer:e], cur)
            if layer >= n:
                cur.wait_event(self._merge_ev[layer - n])     # (its workspace is free again)
            ws = self.attn_ws_slots[layer % n]
            q, k, rope = ((self.q_rot[layer], self.k_rot[layer], None) if self.prerotate
                          else (i.q[layer], i.k_new[layer], self.rope))
            gv.gv_verify_attention_split(self.shape, q, k, i.v_new[layer], i.cacheK[layer], i.cacheV[layer],
                                         i.prefix_len, rope, self.anc, self.treeK[layer], self.treeV[layer],
                                         self.attn_out[layer], ws, cur)
            self._split_ev[layer].record(cur)
            side.wait_event(self._split_ev[layer])
            gv.gv_verify_attention_merge(self.shape, self.attn_out[layer], ws, side)
            self._merge_ev[layer].record(side)

    def join_merges(self, stream=None):
        if self.layers_call:
            return    # (no merges on a second stream)
        cur = stream if stream is not None else torch.cuda.current_stream()
        cur.wait_stream(self.merge_stream)

    def lmhead(self, stream=None):
        i = self.inp
        gv.gv_lmhead_select(i.h, i.W, self.lm_mode, 1, self.ids, self.vals, self.logits,
                            self.row_max, self.row_lse, self.lm_ws, stream)

    def accept(self, stream=None):
        i = self.inp
        B, N, V = self.cfg["B"], self.cfg["N"], self.cfg["V"]
        if self.T == 0.0:
            gv.gv_accept(self.cfg["D"], 0.0, i.tokens, self.anc, self.depth, self.ids, None, None,
                         None, None, self.path, self.accept_len, self.out_tokens, self.seq_status,
                         None, V, stream)
        else:
            gv.gv_accept(self.cfg["D"], self.T, i.tokens, self.anc, self.depth, None,
                         self.logits.view(B, N, V), i.draft_logits, i.u_acc, i.u_res, self.path,
                         self.accept_len, self.out_tokens, self.seq_status, self.acc_ws, V, stream)

    def compact(self, stream=None):
        i = self.inp
        L = self.cfg["L"]
        gv.gv_kv_compact(self.cfg["D"], self.treeK, self.treeV, i.cacheK[:L], i.cacheV[:L],
                         self.path, self.accept_len, i.prefix_len, self.new_len, self.seq_status,
                         stream)

    def run(self, stream=None):
        self.tree(stream)
        self.attention_layers(stream)
        self.lmhead(stream)
        self.accept(stream)
        self.compact(stream)
        self.join_merges(stream)

    # -------------------------------------------------------------- graphs --
    def capture(self):
        """Capture ``run`` into a CUDA graph (after one eager warm-up run)."""
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.run(s)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run(torch.cuda.current_stream())
        self.graph = g
        return g

    def replay(self):
        self.graph.replay()

    # ------------------------------------------------ steps fed from the host --
    # Per-layer inputs a layer waits for, grouped so that each group's copies
    # finish before the compute reaches it.  Per-layer attention: the first
    # layers wait for their own copies, later groups double in size (the
    # copies run ahead of the attention layers, which take several times
    # longer than one layer's copy).  Multi-layer attention (one call per
    # group, each with its own fixed cost): two groups, the first about 28 %
    # of the layers, so that the rest's copy (about 3.6 us a layer at the
    # measured 207 GB/s) lands while the first group's attention (about
    # 5.4 us a layer plus a call's fixed cost) runs.
    COPY_GROUP_CAP = 0    # largest group (layers, per-layer attention); 0: no cap
    LAYERS_CALL_FIRST = 0.28

    def _copy_groups(self, L):
        if self.layers_call:
            k = max(1, min(L, math.ceil(self.LAYERS_CALL_FIRST * L)))
            return [(0, k)] + ([(k, L)] if k < L else [])
        out, a, size = [], 0, 1
        while a < L:
            b = min(L, a + size)
            out.append((a, b))
            a = b
            size = 2 * size if self.COPY_GROUP_CAP <= 0 else min(self.COPY_GROUP_CAP, 2 * size)
        return out

    HOST_INPUTS = ("parents", "tokens", "prefix_len", "qkv", "h", "draft_logits", "u_acc", "u_res")

    def host_buffers(self):
        """Pinned host buffers for a host-fed step, filled from the current
        device inputs: the caller writes each step's inputs into them before
        the replay of ``capture_from_host``'s graph.  The per-layer q, k_new
        and v_new are packed as ``qkv[L][q | k_new | v_new]`` (one copy per
        group of layers); the step's device q, k_new and v_new become views
        of a device buffer with the same layout.  Returns (inputs by name,
        result buffer shaped like ``self.result``)."""
        i = self.inp
        L = self.cfg["L"]
        nq, nk = i.q[0].numel(), i.k_new[0].numel()
        qkv = torch.empty(L, nq + 2 * nk, dtype=i.q.dtype, device=i.q.device)
        qkv[:, :nq].copy_(i.q.reshape(L, nq))
        qkv[:, nq:nq + nk].copy_(i.k_new.reshape(L, nk))
        qkv[:, nq + nk:].copy_(i.v_new.reshape(L, nk))
        i.q = qkv[:, :nq].view(i.q.shape)
        i.k_new = qkv[:, nq:nq + nk].view(i.k_new.shape)
        i.v_new = qkv[:, nq + nk:].view(i.v_new.shape)
        self.qkv = qkv
        host = {"qkv": qkv.cpu().pin_memory()}
        for n in self.HOST_INPUTS:
            if n != "qkv" and getattr(i, n) is not None:
                host[n] = getattr(i, n).cpu().pin_memory()
        out = torch.empty(self.result.shape, dtype=self.result.dtype, pin_memory=True)
        return host, out

    def run_from_host(self, host, host_out, stream, copy_stream):
        """The step with its inputs copied from the pinned buffers of
        ``host_buffers`` and its result (``self.result``: accept_len,
        out_tokens, path) copied back to ``host_out``.  The tree inputs are
        copied on ``stream`` before the tree build; the packed per-layer
        q, k_new, v_new, then the tokens, hidden states and sampling inputs on
        ``copy_stream`` after them, so that they stream in while the earlier
        layers run."""
        i = self.inp
        L = self.cfg["L"]
        # The tree inputs first: the copy engine serves copies in order, so
        # the per-layer copies are queued only after them.
        with torch.cuda.stream(stream):
            for n in ("parents", "prefix_len"):
                getattr(i, n).copy_(host[n], non_blocking=True)
        copy_stream.wait_stream(stream)
        groups = self._copy_groups(L)
        ready = []
        with torch.cuda.stream(copy_stream):
            for a, b in groups:
                self.qkv[a:b].copy_(host["qkv"][a:b], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(copy_stream)
                ready.append(ev)
            for n in ("tokens", "h", "draft_logits", "u_acc", "u_res"):
                if getattr(i, n) is not None and n in host:
                    getattr(i, n).copy_(host[n], non_blocking=True)
            late = torch.cuda.Event()
            late.record(copy_stream)
        self.tree(stream)
        first = {a: ev for (a, _), ev in zip(groups, ready)}
        self.attention_layers(stream, ready=first)
        stream.wait_event(late)
        self.lmhead(stream)
        self.accept(stream)
        self.compact(stream)
        with torch.cuda.stream(stream):
            host_out.copy_(self.result, non_blocking=True)
        self.join_merges(stream)

    def capture_from_host(self, host, host_out):
        """Capture ``run_from_host`` into a CUDA graph (after one eager run)
        over the buffers ``host_buffers`` returned."""
        main, side = torch.cuda.Stream(), torch.cuda.Stream()
        main.wait_stream(torch.cuda.current_stream())
        self.run_from_host(host, host_out, main, side)
        main.wait_stream(side)
        torch.cuda.current_stream().wait_stream(main)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=main):
            self.run_from_host(host, host_out, main, side)
            main.wait_stream(side)
        self.host_graph = g
        return g
