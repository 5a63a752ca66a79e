"""ctypes binding of libgv.so: the C-ABI calls of include/gv.h under the same
names, taking torch CUDA tensors.

This layer only marshals arguments (device pointers, sizes, the current
stream); every step of the verify pass runs in the library's CUDA kernels.
There is no fallback: if libgv.so is missing, or a tensor is not on a CUDA
device, the calls raise.
"""

import ctypes
import os

import torch

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libgv.so")

GV_OK = 0
GV_ERR_ARG = -1
GV_ERR_INVALID_TREE = -2
GV_ERR_CAPACITY = -3
GV_ERR_UNSUPPORTED = -4
GV_ERR_CUDA = -5
GV_ERR_TIMEOUT = -6

GV_BF16 = 0
GV_F32 = 1

GV_SELECT_ARGMAX = 0
GV_SELECT_TOPK = 1
GV_SELECT_LOGITS = 2
GV_LINEAR_STORE, GV_LINEAR_ADD, GV_LINEAR_SWIGLU, GV_LINEAR_SILU = 0, 1, 2, 3

# Every symbol include/gv.h declares.
EXPORTS = ("gv_tree_build", "gv_rope_table", "gv_verify_attention_workspace", "gv_verify_attention",
           "gv_verify_attention_split", "gv_verify_attention_merge", "gv_rope_apply",
           "gv_verify_attention_layers_workspace", "gv_verify_attention_layers",
           "gv_lmhead_workspace", "gv_lmhead_select", "gv_lmhead_argmax_noalloc",
           "gv_accept_workspace", "gv_accept",
           "gv_kv_compact", "gv_rmsnorm", "gv_linear_workspace", "gv_linear", "gv_linear_qkv_workspace",
           "gv_linear_qkv", "gv_linear_add_rmsnorm", "gv_tat_loss", "gv_tgf_workspace", "gv_tgf",
           "gv_draft_tree_workspace", "gv_draft_tree_expand", "gv_draft_tree_finish",
           "gv_status_string", "gv_last_error", "gv_version")


class GvError(RuntimeError):
    def __init__(self, call, status, detail):
        super().__init__(f"{call} -> {status_string(status)} ({status}): {detail}")
        self.status = status


class gv_attn_shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("N", ctypes.c_int), ("Hq", ctypes.c_int),
                ("Hkv", ctypes.c_int), ("d", ctypes.c_int), ("S_max", ctypes.c_int),
                ("dt", ctypes.c_int)]


_lib = None
_vp = ctypes.c_void_p
_i = ctypes.c_int
_f = ctypes.c_float
_sz = ctypes.c_size_t
_i64 = ctypes.c_int64


def lib():
    """Load libgv.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -m paper_2502_11018_gb300.build` (nvcc, sm_103a)")
    L = ctypes.CDLL(LIB_PATH)
    sig = {
        "gv_tree_build": ([_vp, _vp, _i, _i, _vp, _vp, _vp, _vp, _vp], _i),
        "gv_rope_table": ([_vp, _i, _i, _i, _f, _vp, _vp], _i),
        "gv_verify_attention_workspace": ([ctypes.POINTER(gv_attn_shape)], _sz),
        "gv_verify_attention": ([ctypes.POINTER(gv_attn_shape)] + [_vp] * 12 + [_sz, _vp], _i),
        "gv_verify_attention_split": ([ctypes.POINTER(gv_attn_shape)] + [_vp] * 12 + [_sz, _vp], _i),
        "gv_verify_attention_merge": ([ctypes.POINTER(gv_attn_shape), _vp, _vp, _sz, _vp], _i),
        "gv_rope_apply": ([ctypes.POINTER(gv_attn_shape), _i, _vp, _sz, _vp, _sz, _vp, _vp, _vp, _vp], _i),
        "gv_verify_attention_layers_workspace": ([ctypes.POINTER(gv_attn_shape), _i], _sz),
        "gv_verify_attention_layers": ([ctypes.POINTER(gv_attn_shape), _i, _vp, _i64, _vp, _i64, _vp, _i64,
                                        _vp, _vp, _i64] + [_vp] * 7 + [_sz, _vp], _i),
        "gv_lmhead_workspace": ([_i, _i, _i, _i, _i, _i], _sz),
        "gv_lmhead_select": ([_vp, _vp, _i, _i, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp, _vp,
                              _sz, _vp], _i),
        "gv_lmhead_argmax_noalloc": ([_vp, _vp, _i, _i, _i, _vp, _vp, _vp], _i),
        "gv_accept_workspace": ([_i, _i, _f], _sz),
        "gv_accept": ([_i, _i, _i, _i, _f] + [_vp] * 12 + [_vp, _sz, _vp], _i),
        "gv_kv_compact": ([_i] * 8 + [_vp] * 9 + [_vp], _i),
        "gv_rmsnorm": ([_vp, _vp, _i, _i, _f, _vp, _vp], _i),
        "gv_linear_workspace": ([_i, _i, _i, _i], _sz),
        "gv_linear": ([_vp, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _sz, _vp], _i),
        "gv_linear_qkv_workspace": ([_i, _i, _i, _i], _sz),
        "gv_linear_qkv": ([_vp, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _sz, _vp], _i),
        "gv_linear_add_rmsnorm": ([_vp, _vp, _i, _i, _i, _vp, _vp, _vp, _f, _vp, _vp, _sz, _vp], _i),
        "gv_tat_loss": ([_vp, _i, _vp, _vp, _vp, _i, _i, _i, _i, _i, _i, _i, _vp, _f, _f,
                         _vp, _vp, _vp, _vp, _vp], _i),
        "gv_tgf_workspace": ([_i, _i, _i], _sz),
        "gv_draft_tree_workspace": ([_i, _i, _i, _i], _sz),
        "gv_draft_tree_expand": ([_i] * 6 + [_vp] * 5 + [_sz, _vp], _i),
        "gv_draft_tree_finish": ([_i] * 5 + [_vp] * 3 + [_sz, _vp], _i),
        "gv_tgf": ([_vp, _vp, _i, _i, _i] + [_vp] * 10 + [_f, _vp, _vp, _vp, _sz, _vp], _i),
        "gv_status_string": ([_i], ctypes.c_char_p),
        "gv_last_error": ([], ctypes.c_char_p),
        "gv_version": ([], _i),
    }
    for name, (args, res) in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = res
    _lib = L
    return L


def status_string(status):
    return lib().gv_status_string(int(status)).decode()


def last_error():
    return lib().gv_last_error().decode()


def _check(call, rc):
    if rc != GV_OK:
        raise GvError(call, rc, last_error())
    return rc


def _ptr(t, name):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch tensor")
    if not t.is_cuda:
        raise ValueError(f"{name}: tensor must live on a CUDA device (no CPU path)")
    if not t.is_contiguous():
        raise ValueError(f"{name}: tensor must be contiguous")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def dtype_code(t):
    if t.dtype == torch.bfloat16:
        return GV_BF16
    if t.dtype == torch.float32:
        return GV_F32
    raise ValueError(f"unsupported dtype {t.dtype}")


# ------------------------------------------------------------------- calls --

def gv_tree_build(parents, prefix_len, depth, pos, anc, seq_status, stream=None):
    B, N = parents.shape
    return _check("gv_tree_build", lib().gv_tree_build(
        _ptr(parents, "parents"), _ptr(prefix_len, "prefix_len"), B, N, _ptr(depth, "depth"),
        _ptr(pos, "pos"), _ptr(anc, "anc"), _ptr(seq_status, "seq_status"), _stream(stream)))


def gv_rope_table(pos, d, rope_base, rope, stream=None):
    B, N = pos.shape
    return _check("gv_rope_table", lib().gv_rope_table(
        _ptr(pos, "pos"), B, N, d, float(rope_base), _ptr(rope, "rope"), _stream(stream)))


def attn_shape(B, N, Hq, Hkv, d, S_max, dt):
    return gv_attn_shape(B, N, Hq, Hkv, d, S_max, int(dt))


def gv_verify_attention_workspace(shape):
    return int(lib().gv_verify_attention_workspace(ctypes.byref(shape)))


def gv_verify_attention_split(shape, q, k_new, v_new, cacheK, cacheV, prefix_len, rope, anc, treeK,
                              treeV, out, workspace, stream=None):
    """The key-split half of gv_verify_attention (see include/gv.h)."""
    return _check("gv_verify_attention_split", lib().gv_verify_attention_split(
        ctypes.byref(shape), _ptr(q, "q"), _ptr(k_new, "k_new"), _ptr(v_new, "v_new"),
        _ptr(cacheK, "cacheK"), _ptr(cacheV, "cacheV"), _ptr(prefix_len, "prefix_len"),
        _ptr(rope, "rope"), _ptr(anc, "anc"), _ptr(treeK, "treeK"), _ptr(treeV, "treeV"),
        _ptr(out, "out"), _ptr(workspace, "workspace"), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def gv_rope_apply(shape, q, k_new, rope, q_out, k_out, stream=None):
    """Rotate L layers' tree queries and keys (see include/gv.h): q [L][B][N][Hq][d]
    and k_new [L][B][N][Hkv][d], each layer contiguous (any layer stride, e.g.
    views of a packed per-layer buffer); outputs packed."""
    L = q.shape[0]

    def layered(t, name):
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t[0].is_contiguous()):
            raise ValueError(f"{name}: CUDA tensor whose layers are contiguous expected")
        return ctypes.c_void_p(t.data_ptr()), (t.stride(0) if L > 1 else t[0].numel())

    qp, qs = layered(q, "q")
    kp, ks = layered(k_new, "k_new")
    return _check("gv_rope_apply", lib().gv_rope_apply(
        ctypes.byref(shape), L, qp, qs, kp, ks, _ptr(rope, "rope"), _ptr(q_out, "q_out"), _ptr(k_out, "k_out"),
        _stream(stream)))


def gv_verify_attention_merge(shape, out, workspace, stream=None):
    """The merge half of gv_verify_attention (see include/gv.h)."""
    return _check("gv_verify_attention_merge", lib().gv_verify_attention_merge(
        ctypes.byref(shape), _ptr(out, "out"), _ptr(workspace, "workspace"),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def gv_verify_attention(shape, q, k_new, v_new, cacheK, cacheV, prefix_len, rope, anc, treeK,
                        treeV, out, workspace, stream=None):
    return _check("gv_verify_attention", lib().gv_verify_attention(
        ctypes.byref(shape), _ptr(q, "q"), _ptr(k_new, "k_new"), _ptr(v_new, "v_new"),
        _ptr(cacheK, "cacheK"), _ptr(cacheV, "cacheV"), _ptr(prefix_len, "prefix_len"),
        _ptr(rope, "rope"), _ptr(anc, "anc"), _ptr(treeK, "treeK"), _ptr(treeV, "treeV"),
        _ptr(out, "out"), _ptr(workspace, "workspace"), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def gv_verify_attention_layers_workspace(shape, L):
    return int(lib().gv_verify_attention_layers_workspace(ctypes.byref(shape), int(L)))


def _layered(t, name, L):
    """(pointer, layer stride in elements) of a [L][...] CUDA tensor whose
    layers are each contiguous (any layer stride, e.g. views of a packed
    per-layer buffer)."""
    if not (isinstance(t, torch.Tensor) and t.is_cuda and t[0].is_contiguous()):
        raise ValueError(f"{name}: CUDA tensor whose layers are contiguous expected")
    return ctypes.c_void_p(t.data_ptr()), (t.stride(0) if L > 1 else t[0].numel())


def gv_verify_attention_layers(shape, q, k_new, v_new, cacheK, cacheV, prefix_len, rope, anc, treeK, treeV,
                               out, workspace, stream=None):
    """The attention of L layers in one call (see include/gv.h): q, k_new,
    v_new, cacheK, cacheV are [L][...] with contiguous layers; treeK, treeV
    and out packed [L][...]."""
    L = q.shape[0]
    qp, qs = _layered(q, "q", L)
    kp, ks = _layered(k_new, "k_new", L)
    vp, vs = _layered(v_new, "v_new", L)
    ckp, cs = _layered(cacheK, "cacheK", L)
    cvp, cs2 = _layered(cacheV, "cacheV", L)
    if cs != cs2:
        raise ValueError("cacheK and cacheV need the same layer stride")
    return _check("gv_verify_attention_layers", lib().gv_verify_attention_layers(
        ctypes.byref(shape), L, qp, qs, kp, ks, vp, vs, ckp, cvp, cs, _ptr(prefix_len, "prefix_len"),
        _ptr(rope, "rope"), _ptr(anc, "anc"), _ptr(treeK, "treeK"), _ptr(treeV, "treeV"), _ptr(out, "out"),
        _ptr(workspace, "workspace"), workspace.numel() * workspace.element_size(), _stream(stream)))


def gv_lmhead_workspace(rows, H, V, dt, mode, k=1):
    return int(lib().gv_lmhead_workspace(rows, H, V, dt, mode, k))


def gv_lmhead_select(h, W, mode, k, ids, vals, logits, row_max, row_lse, workspace, stream=None):
    rows, H = h.shape
    V = W.shape[0]
    return _check("gv_lmhead_select", lib().gv_lmhead_select(
        _ptr(h, "h"), _ptr(W, "W"), rows, H, V, dtype_code(h), mode, k, _ptr(ids, "ids"),
        _ptr(vals, "vals"), _ptr(logits, "logits"), _ptr(row_max, "row_max"),
        _ptr(row_lse, "row_lse"), _ptr(workspace, "workspace"),
        workspace.numel() * workspace.element_size(), _stream(stream)))


GV_NOALLOC_MAX_ROWS = 256


def gv_lmhead_argmax_noalloc(h, W, ids, vals=None, stream=None):
    """Argmax LM head (bf16) that takes no workspace: its scratch is a fixed
    array inside the library (rows <= GV_NOALLOC_MAX_ROWS; calls that overlap
    in time on one device race)."""
    rows, H = h.shape
    V = W.shape[0]
    return _check("gv_lmhead_argmax_noalloc", lib().gv_lmhead_argmax_noalloc(
        _ptr(h, "h"), _ptr(W, "W"), rows, H, V, _ptr(ids, "ids"), _ptr(vals, "vals"),
        _stream(stream)))


def gv_accept_workspace(B, V, temperature):
    return int(lib().gv_accept_workspace(B, V, float(temperature)))


def gv_accept(D, temperature, tokens, anc, depth, choice, target_logits, draft_logits, u_acc,
              u_res, path, accept_len, out_tokens, seq_status, workspace=None, V=0, stream=None):
    B, N = tokens.shape
    if target_logits is not None:
        V = target_logits.shape[-1]
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    return _check("gv_accept", lib().gv_accept(
        B, N, D, V, float(temperature), _ptr(tokens, "tokens"), _ptr(anc, "anc"),
        _ptr(depth, "depth"), _ptr(choice, "choice"), _ptr(target_logits, "target_logits"),
        _ptr(draft_logits, "draft_logits"), _ptr(u_acc, "u_acc"), _ptr(u_res, "u_res"),
        _ptr(path, "path"), _ptr(accept_len, "accept_len"), _ptr(out_tokens, "out_tokens"),
        _ptr(seq_status, "seq_status"), _ptr(workspace, "workspace"), ws_bytes, _stream(stream)))


def gv_kv_compact(D, treeK, treeV, cacheK, cacheV, path, accept_len, prefix_len, new_len,
                  seq_status, stream=None):
    L, B, Hkv, N, d = treeK.shape
    S_max = cacheK.shape[3]
    return _check("gv_kv_compact", lib().gv_kv_compact(
        L, B, N, D, Hkv, d, S_max, dtype_code(treeK), _ptr(treeK, "treeK"), _ptr(treeV, "treeV"),
        _ptr(cacheK, "cacheK"), _ptr(cacheV, "cacheV"), _ptr(path, "path"),
        _ptr(accept_len, "accept_len"), _ptr(prefix_len, "prefix_len"), _ptr(new_len, "new_len"),
        _ptr(seq_status, "seq_status"), _stream(stream)))


def gv_tat_loss(logits, tokens, feat_draft, feat_target, k, n, mbar_prev, mbar, mask, ell, seq_loss,
                lambda_tok=1.0, lambda_feat=0.1, stream=None):
    """One token-alignable training pass (see include/gv.h).  logits [B][T][V],
    tokens int32 [B][T], features [B][T][H], mbar_prev uint8 [n-1][B][T] or
    None (n == 1); outputs mbar, mask uint8 [B][T], ell fp32 [B][T],
    seq_loss fp32 [B]."""
    B, T, V = logits.shape
    H = feat_draft.shape[2]
    return _check("gv_tat_loss", lib().gv_tat_loss(
        _ptr(logits, "logits"), dtype_code(logits), _ptr(tokens, "tokens"), _ptr(feat_draft, "feat_draft"),
        _ptr(feat_target, "feat_target"), dtype_code(feat_draft), B, T, V, H, k, n,
        _ptr(mbar_prev, "mbar_prev"), float(lambda_tok), float(lambda_feat), _ptr(mbar, "mbar"),
        _ptr(mask, "mask"), _ptr(ell, "ell"), _ptr(seq_loss, "seq_loss"), _stream(stream)))


def gv_tgf_workspace(rows, d, e):
    return int(lib().gv_tgf_workspace(rows, d, e))


def gv_tgf(F, x, w, h_out, o_out, workspace, eps=1e-5, stream=None):
    """Token-Guided Fusion (see include/gv.h): F, x [rows][d]; ``w`` maps Wm,
    bm, g_h, b_h, g_x, b_x, Wu, bu, Wd, bd to bf16 tensors; outputs h_out and
    o_out [rows][d]."""
    rows, d = F.shape
    e = w["Wu"].shape[0]
    ws_bytes = workspace.numel() * workspace.element_size()
    names = ("Wm", "bm", "g_h", "b_h", "g_x", "b_x", "Wu", "bu", "Wd", "bd")
    return _check("gv_tgf", lib().gv_tgf(
        _ptr(F, "F"), _ptr(x, "x"), rows, d, e, *[_ptr(w[n], n) for n in names], float(eps),
        _ptr(h_out, "h_out"), _ptr(o_out, "o_out"), _ptr(workspace, "workspace"), ws_bytes, _stream(stream)))


def gv_draft_tree_workspace(B, k, D, V):
    return int(lib().gv_draft_tree_workspace(B, k, D, V))


def gv_draft_tree_expand(step, k, D, logits, workspace, root_token=None, exp_token=None, exp_pool=None,
                         stream=None):
    """One expansion step of the draft tree (see include/gv.h): logits
    [B][rows][V] (rows = 1 at step 0, else k), fp32 or bf16."""
    B, _, V = logits.shape
    ws_bytes = workspace.numel() * workspace.element_size()
    return _check("gv_draft_tree_expand", lib().gv_draft_tree_expand(
        B, k, D, V, step, dtype_code(logits), _ptr(root_token, "root_token"), _ptr(logits, "logits"),
        _ptr(exp_token, "exp_token"), _ptr(exp_pool, "exp_pool"), _ptr(workspace, "workspace"), ws_bytes,
        _stream(stream)))


def gv_draft_tree_finish(k, D, V, parents, tokens, workspace, stream=None):
    """The rerank: parents, tokens int32 [B][N] of the tree (see include/gv.h)."""
    B, N = parents.shape
    ws_bytes = workspace.numel() * workspace.element_size()
    return _check("gv_draft_tree_finish", lib().gv_draft_tree_finish(
        B, k, D, V, N, _ptr(parents, "parents"), _ptr(tokens, "tokens"), _ptr(workspace, "workspace"), ws_bytes,
        _stream(stream)))


def gv_rmsnorm(x, w, out, eps=1e-5, stream=None):
    """RMSNorm of the rows of x [rows][H] with weight w [H] into out (bf16)."""
    rows, H = x.shape
    return _check("gv_rmsnorm", lib().gv_rmsnorm(_ptr(x, "x"), _ptr(w, "w"), rows, H, float(eps),
                                                 _ptr(out, "out"), _stream(stream)))


def gv_linear_workspace(rows, K, n_out, epilogue=0):
    return int(lib().gv_linear_workspace(rows, K, n_out, epilogue))


def gv_linear(x, W, out, epilogue=0, residual=None, workspace=None, stream=None):
    """out [rows][n_out] = epilogue(x W^T) (see include/gv.h)."""
    rows, K = x.shape
    n_out = out.shape[1]
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    return _check("gv_linear", lib().gv_linear(
        _ptr(x, "x"), _ptr(W, "W"), rows, K, n_out, int(epilogue), _ptr(residual, "residual"), _ptr(out, "out"),
        _ptr(workspace, "workspace"), ws_bytes, _stream(stream)))


def gv_linear_qkv_workspace(rows, K, n_q, n_kv):
    return int(lib().gv_linear_qkv_workspace(rows, K, n_q, n_kv))


def gv_linear_qkv(x, Wqkv, q, k, v, workspace, stream=None):
    """q, k, v = x [Wq ; Wk ; Wv]^T, one weight stream (see include/gv.h)."""
    rows, K = x.shape
    n_q = q.numel() // rows
    n_kv = k.numel() // rows
    ws_bytes = workspace.numel() * workspace.element_size()
    return _check("gv_linear_qkv", lib().gv_linear_qkv(
        _ptr(x, "x"), _ptr(Wqkv, "Wqkv"), rows, K, n_q, n_kv, _ptr(q, "q"), _ptr(k, "k"), _ptr(v, "v"),
        _ptr(workspace, "workspace"), ws_bytes, _stream(stream)))


def gv_linear_add_rmsnorm(x, W, residual, out, norm_w, norm_out, workspace, eps=1e-5, stream=None):
    """out = residual + x W^T, norm_out = RMSNorm(out) * norm_w (see include/gv.h)."""
    rows, K = x.shape
    n_out = out.shape[1]
    ws_bytes = workspace.numel() * workspace.element_size()
    return _check("gv_linear_add_rmsnorm", lib().gv_linear_add_rmsnorm(
        _ptr(x, "x"), _ptr(W, "W"), rows, K, n_out, _ptr(residual, "residual"), _ptr(out, "out"),
        _ptr(norm_w, "norm_w"), float(eps), _ptr(norm_out, "norm_out"), _ptr(workspace, "workspace"), ws_bytes,
        _stream(stream)))
