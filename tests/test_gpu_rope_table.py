"""GPU check of gv_rope_table against cos and sin of the float64 angle
pos * base^(-2j/d), the angle the oracle's rotation uses: every entry within
3e-7 (absolute) of the float64 values, over positions up to 2^24 (so the
reduction modulo 2 pi is exercised far past the prefixes of the workloads),
head dims 2 .. 256 and RoPE bases 1e4 .. 1e6."""

import numpy as np
import pytest
import torch

from gpu_util import device

from paper_2502_11018_gb300 import gv

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("d,base", [(128, 5e5), (64, 1e4), (256, 1e6), (2, 1e4), (128, 1e4)])
def test_rope_table_matches_float64(d, base):
    dev = device()
    rng = np.random.default_rng(d)
    B, N = 3, 64
    pos = rng.integers(0, 1 << 24, size=(B, N)).astype(np.int32)
    pos[0, :8] = [0, 1, 2, 4095, 4096, 4155, 16383, 1 << 20]
    pos_d = torch.as_tensor(pos, device=dev)
    rope = torch.full((B, N, d // 2, 2), float("nan"), dtype=torch.float32, device=dev)
    gv.gv_rope_table(pos_d, d, base, rope)
    torch.cuda.synchronize()
    got = rope.cpu().double().numpy()
    j = np.arange(d // 2, dtype=np.float64)
    ang = pos.astype(np.float64)[..., None] * np.power(float(np.float32(base)), -2.0 * j / d)
    assert np.abs(got[..., 0] - np.cos(ang)).max() <= 3e-7
    assert np.abs(got[..., 1] - np.sin(ang)).max() <= 3e-7
