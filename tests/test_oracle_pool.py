"""Pins of the oracle's super-sampled position maps (Sec. 3.1: position maps
are rendered at image resolution; Sec. 3.2: the correspondence operator acts
on the latent token grid).  A token's position is the mean of its valid
sub-pixels' positions and it is foreground when at least half of them are
valid; the checks below tie that to closed forms rather than to the oracle's
own arithmetic."""
import numpy as np
import pytest

import oracle
from paper_2608_13255_gb300 import synth


def test_factor_one_is_the_identity():
    w = synth.make_workload("hunyuan64", H=32, W=32)
    pos, valid = w.pos[0], w.valid[0]
    p1, v1 = oracle.pool(pos, valid, 1)
    np.testing.assert_array_equal(v1, valid)
    np.testing.assert_array_equal(p1, np.where(valid[..., None] > 0, pos, 0.0).astype(np.float32))


@pytest.mark.parametrize("s", [2, 4, 8])
def test_camera_aligned_plane_pools_to_the_token_centres(s):
    # the fine map of a fronto-parallel plane is affine in the pixel
    # coordinates, so the mean over a token's s x s sub-pixel centres is the
    # position at the token centre: the coarse map of the same plane, exactly
    H, W, f = 24, 40, 64.0
    _, fine, fine_valid = synth.camera_aligned_plane(H * s, W * s, focal=f * s, radius_frac=10.0)
    _, coarse, coarse_valid = synth.camera_aligned_plane(H, W, focal=f, radius_frac=10.0)
    assert fine_valid.all() and coarse_valid.all()
    p, v = oracle.pool(fine, fine_valid, s)
    assert v.all()
    np.testing.assert_array_equal(p, coarse)


@pytest.mark.parametrize("s", [2, 3, 4, 8])
def test_validity_is_at_least_half_and_position_is_the_mean_of_the_valid(s):
    # tokens with every possible number c of valid sub-pixels (random
    # positions, random placement): foreground iff 2 c >= s^2, position the
    # mean of exactly those sub-pixels
    rng = np.random.default_rng(s)
    n_tok = s * s + 1
    H, W = 1, n_tok
    fine = rng.uniform(-2, 2, (H * s, W * s, 3)).astype(np.float32)
    fine_valid = np.zeros((H * s, W * s), np.uint8)
    for i in range(W):
        cells = rng.permutation(s * s)[:i]  # token i has exactly i valid sub-pixels
        fine_valid[cells // s, i * s + cells % s] = 1
    p, v = oracle.pool(fine, fine_valid, s)
    for i in range(W):
        blk = fine[:, i * s:(i + 1) * s].reshape(-1, 3).astype(np.float64)
        m = fine_valid[:, i * s:(i + 1) * s].reshape(-1) > 0
        assert v[0, i] == (2 * m.sum() >= s * s)
        if v[0, i]:
            np.testing.assert_allclose(p[0, i], blk[m].mean(0), rtol=0, atol=4e-7 * m.sum())
        else:
            assert (p[0, i] == 0).all()


def _quad(x0, x1, y0, y1, z):
    V = np.array([[x0, y0, z], [x1, y0, z], [x1, y1, z], [x0, y1, z]], np.float32)
    F = np.array([[0, 1, 2], [0, 2, 3]], np.int32)
    return V, F


@pytest.mark.parametrize("s", [4, 8])
def test_rendered_rectangle_keeps_the_tokens_it_covers_at_least_half(s):
    # a camera-aligned rectangle whose edges cut tokens at 5/8 and 3/8 of
    # their width, rendered at s x the token grid: a token is foreground when
    # the sub-pixel centres inside or on the rectangle (columns x rows) are
    # at least half of its s x s; fully covered tokens pool to the
    # closed-form position at the token centre
    H = W = 32
    f, depth = 64.0, 4.0
    cam = synth.camera_aligned_plane(H, W, focal=f, depth=depth)[0]
    lo, hi = 10 + 5 / 8, 20 + 3 / 8  # token units
    to_world = lambda u, c: (u - c) * depth / f
    V, F = _quad(to_world(lo, W / 2), to_world(hi, W / 2), to_world(lo, H / 2), to_world(hi, H / 2), depth / 2)
    pos, valid = oracle.raster_supersampled(V, F, cam[None], H, W, s)
    centres = (np.arange(s) + 0.5) / s
    cover = np.zeros(W, np.int64)  # covered sub-pixel columns (= rows) of each token
    for t in range(W):
        cover[t] = ((t + centres >= lo) & (t + centres <= hi)).sum()
    expect = (2 * cover[:, None] * cover[None, :] >= s * s).astype(np.uint8)
    assert expect[11:20, 11:20].all() and not expect[:10].any() and not expect[21:].any()
    np.testing.assert_array_equal(valid[0], expect)
    full = cover[:, None] * cover[None, :] == s * s
    _, plane, _ = synth.camera_aligned_plane(H, W, focal=f, depth=depth, radius_frac=10.0)
    np.testing.assert_allclose(pos[0][full], plane[full], rtol=0, atol=1e-6)
    # the fine render itself covers exactly those sub-pixel columns
    fp, fv = oracle.raster(V, F, oracle.scaled_camera(cam, s), H * s, W * s)
    assert fv[11 * s:20 * s, 10 * s:11 * s].sum() == 9 * s * cover[10]
