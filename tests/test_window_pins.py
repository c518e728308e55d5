"""Pins of the re-anchored audio window (oracle/window.py): geometry from the
paper's stated widths, and the restricted attention against torch's
multi-head attention with the frames outside the window masked."""
import numpy as np
import pytest
import torch

from oracle.window import frames, window, window_center, windowed_attention


def test_geometry_on_the_20_ms_grid():
    assert frames(400) == 20 and frames(500) == 25
    assert window(100, 1500) == (80, 121)            # 41 frames: 400 ms either side
    assert window(5, 1500) == (0, 26)                # clipped at the start
    assert window(1495, 1500) == (1475, 1500)        # and at the end
    assert window_center("anchor", 700, 1500) == 700
    assert window_center("shifted", 700, 1500) == 725
    assert window_center("shifted", 1490, 1500) == 1499     # clipped to the grid
    assert window_center("anchor", -3, 10) == 0


def test_random_centre_is_uniform_and_seeded():
    assert window_center("random", 0, 50, np.random.default_rng(0)) == window_center("random", 0, 50)   # seed 0
    rng = np.random.default_rng(0)
    draws = np.array([window_center("random", 0, 10, rng) for _ in range(20000)])
    counts = np.bincount(draws, minlength=10)
    chi2 = float(((counts - 2000.0) ** 2 / 2000.0).sum())
    assert draws.min() == 0 and draws.max() == 9 and chi2 < 30.0      # 9 dof, p ~ 4e-4


@pytest.mark.parametrize("center,T", [(37, 120), (2, 60), (118, 120)])
def test_windowed_attention_matches_masked_library_attention(center, T):
    rng = np.random.default_rng(center)
    d, H = 64, 4
    q = rng.standard_normal(d)
    K = rng.standard_normal((T, d))
    V = rng.standard_normal((T, d))
    lo, hi = window(center, T)
    got = windowed_attention(q, K, V, H, lo, hi)
    mha = torch.nn.MultiheadAttention(d, H, bias=False, batch_first=True).double()
    with torch.no_grad():
        for w in (mha.in_proj_weight, mha.out_proj.weight):
            w.zero_()
        mha.in_proj_weight[:d] = torch.eye(d)
        mha.in_proj_weight[d:2 * d] = torch.eye(d)
        mha.in_proj_weight[2 * d:] = torch.eye(d)
        mha.out_proj.weight.copy_(torch.eye(d))
        mask = torch.ones(1, T, dtype=torch.bool)
        mask[0, lo:hi] = False                         # True = not attended
        ref, _ = mha(torch.from_numpy(q)[None, None], torch.from_numpy(K)[None], torch.from_numpy(V)[None],
                     key_padding_mask=mask)
    np.testing.assert_allclose(got, ref[0, 0].numpy(), rtol=0, atol=1e-12)
