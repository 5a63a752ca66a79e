"""The C-ABI library loads on a host without a GPU and exports every function
include/gv.h declares; host-side argument checks answer without launching
anything (no GPU is touched by these tests)."""

import ctypes
import os
import re

import pytest

from paper_2502_11018_gb300 import build, gv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return gv.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "gv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gv_[a-z_]+)\s*\(", src)))


def test_exports_match_header(lib):
    names = declared_functions()
    assert len(names) >= 12
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(gv.EXPORTS) == names


def test_status_strings(lib):
    assert gv.status_string(0) == "GV_OK"
    assert gv.status_string(-2) == "GV_ERR_INVALID_TREE"
    assert gv.status_string(-3) == "GV_ERR_CAPACITY"
    assert gv.status_string(123) == "GV_ERR_UNKNOWN"
    assert lib.gv_version() >= 100


def test_host_side_validation(lib):
    nul = None
    # N outside 1..64 is rejected before any device work.
    assert lib.gv_tree_build(nul, nul, 1, 65, nul, nul, nul, nul, nul) == gv.GV_ERR_INVALID_TREE
    assert lib.gv_tree_build(nul, nul, 1, 0, nul, nul, nul, nul, nul) == gv.GV_ERR_INVALID_TREE
    assert lib.gv_tree_build(nul, nul, 1, 4, nul, nul, nul, nul, nul) == gv.GV_ERR_ARG
    assert "null" in gv.last_error()
    shape = gv.attn_shape(1, 60, 32, 8, 96, 4224, gv.GV_BF16)
    assert lib.gv_verify_attention(ctypes.byref(shape), *([nul] * 12), 0, nul) == gv.GV_ERR_UNSUPPORTED
    shape = gv.attn_shape(1, 60, 64, 8, 128, 4224, gv.GV_BF16)   # 480 query rows per KV head
    assert lib.gv_verify_attention(ctypes.byref(shape), *([nul] * 12), 0, nul) == gv.GV_ERR_UNSUPPORTED
    shape = gv.attn_shape(1, 60, 30, 8, 128, 4224, gv.GV_BF16)
    assert gv.gv_verify_attention_workspace(shape) == 0     # Hq not a multiple of Hkv
    assert lib.gv_rope_table(nul, 1, 60, 128, 1e4, nul, nul) == gv.GV_ERR_ARG
    assert lib.gv_lmhead_select(nul, nul, 60, 4096, 1000, 0, 1, 17, *([nul] * 6), 0, nul) == gv.GV_ERR_ARG
    # The allocation-free argmax rejects row counts beyond its fixed scratch.
    assert lib.gv_lmhead_argmax_noalloc(16, 16, gv.GV_NOALLOC_MAX_ROWS + 1, 4096, 1000, 16, nul,
                                        nul) == gv.GV_ERR_UNSUPPORTED
    assert "exceeds the fixed scratch" in gv.last_error()
    assert lib.gv_lmhead_argmax_noalloc(nul, nul, 60, 4096, 1000, nul, nul, nul) == gv.GV_ERR_ARG
    assert lib.gv_accept(1, 60, 6, 0, -1.0, *([nul] * 12), nul, 0, nul) == gv.GV_ERR_ARG
    assert lib.gv_kv_compact(1, 1, 60, 6, 8, 3, 100, 0, *([nul] * 9), nul) == gv.GV_ERR_ARG
    assert "16-byte" in gv.last_error()
    # token-alignable loss: k beyond the vocabulary, mbar_prev given for n = 1
    assert lib.gv_tat_loss(16, gv.GV_F32, 16, 16, 16, gv.GV_BF16, 2, 8, 10, 64, 11, 1, nul, 1.0, 0.1,
                           16, 16, 16, 16, nul) == gv.GV_ERR_ARG
    assert lib.gv_tat_loss(16, gv.GV_F32, 16, 16, 16, gv.GV_BF16, 2, 8, 10, 64, 3, 1, 16, 1.0, 0.1,
                           16, 16, 16, 16, nul) == gv.GV_ERR_ARG
    assert "mbar_prev" in gv.last_error()
    # projections: K not a multiple of 8; a residual without GV_LINEAR_ADD
    assert lib.gv_linear(16, 16, 60, 4100 + 2, 4096, 0, nul, 16, 16, 1 << 30, nul) == gv.GV_ERR_ARG
    assert lib.gv_linear(16, 16, 60, 4096, 4096, 0, 16, 16, 16, 1 << 30, nul) == gv.GV_ERR_ARG
    assert "residual" in gv.last_error()
    assert lib.gv_rmsnorm(16, 16, 60, 4100, 1e-5, 16, nul) == gv.GV_ERR_ARG
    assert gv.gv_linear_workspace(60, 4096, 1024, gv.GV_LINEAR_STORE) > 0
    assert gv.gv_linear_workspace(60, 4096, 14336, gv.GV_LINEAR_SWIGLU) >= 60 * 28672 * 4
    assert gv.gv_linear_workspace(60, 4096, 2048, gv.GV_LINEAR_SILU) > 0
    assert gv.gv_linear_workspace(60, 4096, 2048, 4) == 0
    # token-guided fusion: d not a multiple of 64, rows beyond 256, h_out == o_out
    tgf_w = [16] * 10
    assert lib.gv_tgf(16, 16, 60, 4100, 11008, *tgf_w, 1e-5, 16, 32, 16, 1 << 34, nul) == gv.GV_ERR_ARG
    assert lib.gv_tgf(16, 16, 257, 4096, 11008, *tgf_w, 1e-5, 16, 32, 16, 1 << 34, nul) == gv.GV_ERR_ARG
    assert lib.gv_tgf(16, 16, 60, 4096, 11008, *tgf_w, 1e-5, 16, 16, 16, 1 << 34, nul) == gv.GV_ERR_ARG
    assert "separate" in gv.last_error()
    assert lib.gv_tgf(16, 16, 60, 4096, 11008, *tgf_w, 1e-5, 16, 32, 16, 16, nul) == gv.GV_ERR_ARG
    assert "workspace" in gv.last_error()
    assert gv.gv_tgf_workspace(60, 4096, 11008) >= 60 * (2 * 4096 + 11008) * 2
    assert gv.gv_tgf_workspace(60, 4100, 11008) == 0
    # rotation ahead of the attention: bf16 with d = 128 only; a layer stride below one layer
    f32 = gv.attn_shape(1, 60, 32, 8, 128, 4224, gv.GV_F32)
    assert lib.gv_rope_apply(ctypes.byref(f32), 2, 16, 1 << 20, 16, 1 << 20, 16, 16, 16, nul) == gv.GV_ERR_ARG
    bf = gv.attn_shape(1, 60, 32, 8, 128, 4224, gv.GV_BF16)
    assert lib.gv_rope_apply(ctypes.byref(bf), 2, 16, 64, 16, 1 << 20, 16, 16, 16, nul) == gv.GV_ERR_ARG
    assert "stride" in gv.last_error()
    # draft tree: k beyond 16, a pool beyond 4096 nodes, step out of range, N beyond 64
    assert gv.gv_draft_tree_workspace(1, 17, 6, 32000) == 0
    assert gv.gv_draft_tree_workspace(1, 16, 17, 32000) == 0
    assert gv.gv_draft_tree_workspace(1, 10, 6, 32000) > 0
    assert lib.gv_draft_tree_expand(1, 10, 6, 32000, 6, gv.GV_F32, 16, 16, nul, nul, 16, 1 << 30, nul) == gv.GV_ERR_ARG
    assert "step" in gv.last_error()
    assert lib.gv_draft_tree_expand(1, 10, 6, 32000, 0, gv.GV_F32, nul, 16, nul, nul, 16, 1 << 30, nul) == gv.GV_ERR_ARG
    assert "root_token" in gv.last_error()
    assert lib.gv_draft_tree_finish(1, 10, 6, 32000, 65, 16, 16, 16, 1 << 30, nul) == gv.GV_ERR_ARG


def test_workspace_queries(lib):
    shape = gv.attn_shape(1, 60, 32, 8, 128, 4224, gv.GV_BF16)
    assert gv.gv_verify_attention_workspace(shape) > 0
    assert gv.gv_lmhead_workspace(60, 4096, 128256, gv.GV_BF16, gv.GV_SELECT_ARGMAX) > 0
    assert gv.gv_lmhead_workspace(60, 4096, 128256, gv.GV_BF16, gv.GV_SELECT_TOPK, 0) == 0
    assert gv.gv_accept_workspace(1, 32000, 0.0) == 0
    assert gv.gv_accept_workspace(2, 32000, 1.0) >= 2 * 2 * 32000 * 4
