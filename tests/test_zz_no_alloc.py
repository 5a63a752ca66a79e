"""gv_lmhead_argmax_noalloc (the argmax LM head whose scratch is a fixed array
inside the library) against gv_lmhead_select with a caller workspace, on the
same inputs, for two calls in a row.  The file name sorts last so that the
test also runs after every other GPU test has used the library."""

import pytest
import torch

from paper_2502_11018_gb300 import gv
from gpu_util import device

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("rows,H,V", [(60, 4096, 128256), (256, 1024, 32000), (1, 512, 4100)])
def test_noalloc_argmax_matches_workspace_path(rows, H, V):
    dev = device()
    gen = torch.Generator().manual_seed(rows * 7 + V)
    W = (torch.randn(V, H, generator=gen) * 0.02).to(torch.bfloat16).to(dev)
    # Planted rows: row r points at token t_r, so the argmax is unique by a wide margin.
    t = torch.randint(0, V, (rows,), generator=gen)
    Wt = W.float().cpu()[t]
    h = Wt / Wt.norm(dim=1, keepdim=True) + 0.05 / H ** 0.5 * torch.randn(rows, H, generator=gen)
    h = h.to(torch.bfloat16).to(dev)

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
