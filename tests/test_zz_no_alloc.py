"""gv_lmhead_argmax_noalloc (the argmax LM head whose scratch is a fixed array
inside the library) against gv_lmhead_select with a caller workspace, on the
same inputs, for two calls in a row; and the entry point's promise itself:
a call allocates no device memory (neither PyTorch's allocator nor the
device's free memory moves across it), with vals given or NULL, on the
default stream or a side stream.  The file name sorts last so that the test
also runs after every other GPU test has used the library."""

import pytest
import torch

from paper_2502_11018_gb300 import gv
from gpu_util import device

pytestmark = pytest.mark.gpu


def _planted(rows, H, V, dev):
    gen = torch.Generator().manual_seed(rows * 7 + V)
    W = (torch.randn(V, H, generator=gen) * 0.02).to(torch.bfloat16).to(dev)
    # Planted rows: row r points at token t_r, so the argmax is unique by a wide margin.
    t = torch.randint(0, V, (rows,), generator=gen)
    Wt = W.float().cpu()[t]
    h = Wt / Wt.norm(dim=1, keepdim=True) + 0.05 / H ** 0.5 * torch.randn(rows, H, generator=gen)
    return h.to(torch.bfloat16).to(dev), W, t


def _device_free_bytes():
    free, total = torch.cuda.mem_get_info()
    return free


@pytest.mark.parametrize("rows,H,V", [(60, 4096, 128256), (256, 1024, 32000), (1, 512, 4100)])
def test_noalloc_argmax_matches_workspace_path(rows, H, V):
    dev = device()
    h, W, t = _planted(rows, H, V, dev)
    ws = torch.empty(gv.gv_lmhead_workspace(rows, H, V, gv.GV_BF16, gv.GV_SELECT_ARGMAX),
                     dtype=torch.uint8, device=dev)
    ids_ref = torch.empty(rows, dtype=torch.int32, device=dev)
    vals_ref = torch.empty(rows, dtype=torch.float32, device=dev)
    gv.gv_lmhead_select(h, W, gv.GV_SELECT_ARGMAX, 1, ids_ref, vals_ref, None, None, None, ws)

    for _ in range(2):
        ids = torch.full((rows,), -7, dtype=torch.int32, device=dev)
        vals = torch.full((rows,), float("nan"), dtype=torch.float32, device=dev)
        gv.gv_lmhead_argmax_noalloc(h, W, ids, vals)
        torch.cuda.synchronize()
        assert torch.equal(ids.cpu(), ids_ref.cpu())
        assert torch.equal(ids.cpu(), t.to(torch.int32))
        torch.testing.assert_close(vals.cpu(), vals_ref.cpu(), rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("with_vals,side_stream", [(True, False), (False, True)])
def test_noalloc_call_allocates_nothing(with_vals, side_stream):
    dev = device()
    rows, H, V = 60, 4096, 128256
    h, W, t = _planted(rows, H, V, dev)
    ids = torch.full((rows,), -7, dtype=torch.int32, device=dev)
    vals = torch.full((rows,), float("nan"), dtype=torch.float32, device=dev) if with_vals else None
    stream = torch.cuda.Stream() if side_stream else torch.cuda.current_stream()
    # a first call (the library's kernels and symbols are set up by now)
    with torch.cuda.stream(stream):
        gv.gv_lmhead_argmax_noalloc(h, W, ids, vals, stream=stream)
    torch.cuda.synchronize()
    ids.fill_(-7)
    torch.cuda.synchronize()
    alloc0, free0 = torch.cuda.memory_allocated(), _device_free_bytes()
    with torch.cuda.stream(stream):
        gv.gv_lmhead_argmax_noalloc(h, W, ids, vals, stream=stream)
    torch.cuda.synchronize()
    alloc1, free1 = torch.cuda.memory_allocated(), _device_free_bytes()
    assert alloc1 == alloc0
    assert free1 == free0
    assert torch.equal(ids.cpu(), t.to(torch.int32))
