"""The whole verify forward pass of a LLaMA-style target over a draft tree,
through the C ABI: the decoder layers around the tree attention, then the
final norm, the LM head, acceptance and compaction (GRIFFIN Section 3: one
target forward verifies every draft token).

Per layer, over the hidden states h [B*N][H] of the tree nodes:

    x = RMSNorm(h) * w_attn                      (fused into the previous call)
    q, k, v = x Wq^T, x Wk^T, x Wv^T             gv_linear_qkv (one weight stream)
    o = TreeAttention(q, k, v)                   gv_verify_attention
    h = h + o Wo^T; x = RMSNorm(h) * w_mlp       gv_linear_add_rmsnorm
    g = silu(x Wg^T) * (x Wu^T)                  gv_linear (SwiGLU)
    h = h + g Wd^T; x = RMSNorm(h) * w_next      gv_linear_add_rmsnorm

where w_next is the next layer's w_attn, or after the last layer w_final,
whose output feeds gv_lmhead_select; the first layer's input norm is
gv_rmsnorm of the embeddings.  Nothing here computes: it
owns buffers and issues the calls on one stream (graph-capturable).
"""

import torch

from . import gv
from .step import VerifyStep


class VerifyForward:
    """``inp`` is a ``StepInputs`` (tree, tokens, caches, LM head weight; its
    q / k_new / v_new / h are not used: they are computed here) and ``fw`` a
    ``ForwardWeights`` of matching shapes."""

    def __init__(self, inp, fw):
        self.inp, self.fw = inp, fw
        cfg = inp.cfg
        self.cfg = cfg
        dev = inp.cacheK.device
        B, N, H, Hq, Hkv, d = cfg["B"], cfg["N"], cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["d"]
        R = B * N
        bf = dict(dtype=torch.bfloat16, device=dev)
        self.h = torch.zeros(R, H, **bf)
        self.x = torch.zeros(R, H, **bf)
        self.q = torch.zeros(B, N, Hq, d, **bf)
        self.k = torch.zeros(B, N, Hkv, d, **bf)
        self.v = torch.zeros(B, N, Hkv, d, **bf)
        self.g = torch.zeros(R, fw.F, **bf)
        shapes = [(Hq * d, H, 1), (H, fw.F, 2), (fw.F, H, 1)]
        ws = max([gv.gv_linear_workspace(R, K, n, e) for K, n, e in shapes] +
                 [gv.gv_linear_qkv_workspace(R, H, Hq * d, Hkv * d)])
        self.lin_ws = torch.empty(ws, dtype=torch.uint8, device=dev)
        # The verify step's own buffers (tree, attention outputs, LM head,
        # acceptance); its inputs' q / k_new / v_new / h are bound to ours.
        self.step = VerifyStep(inp)
        self.graph = None

    def _lin(self, x, W, out, epi, residual=None, stream=None):
        gv.gv_linear(x, W, out, epi, residual=residual, workspace=self.lin_ws, stream=stream)

    def layer(self, l, stream=None):
        """Layer l; self.x holds RMSNorm(h) * w_attn[l] on entry."""
        fw, st = self.fw, self.step
        R = self.h.shape[0]
        L = self.cfg["L"]
        h_in = fw.h0 if l == 0 else self.h      # layer 0 reads the embeddings
        gv.gv_linear_qkv(self.x, fw.Wqkv[l], self.q.view(R, -1), self.k.view(R, -1), self.v.view(R, -1),
                         self.lin_ws, stream=stream)
        i = self.inp
        gv.gv_verify_attention(st.shape, self.q, self.k, self.v, i.cacheK[l], i.cacheV[l], i.prefix_len, st.rope,
                               st.anc, st.treeK[l], st.treeV[l], st.attn_out[l], st.attn_ws, stream)
        gv.gv_linear_add_rmsnorm(st.attn_out[l].view(R, -1), fw.Wo[l], h_in, self.h, fw.mlp_norm[l], self.x,
                                 self.lin_ws, stream=stream)
        self._lin(self.x, fw.Wgu[l], self.g, gv.GV_LINEAR_SWIGLU, stream=stream)
        nxt_w, nxt_out = (fw.attn_norm[l + 1], self.x) if l + 1 < L else (fw.final_norm, self.inp.h)
        gv.gv_linear_add_rmsnorm(self.g, fw.Wd[l], self.h, self.h, nxt_w, nxt_out, self.lin_ws, stream=stream)

    def run(self, stream=None):
        """Tree build, every layer, final norm, LM head, acceptance, compaction."""
        st = self.step
        st.tree(stream)
        gv.gv_rmsnorm(self.fw.h0, self.fw.attn_norm[0], self.x, stream=stream)
        for l in range(self.cfg["L"]):
            self.layer(l, stream)
        st.lmhead(stream)
        st.accept(stream)
        st.compact(stream)

    def capture(self):
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
