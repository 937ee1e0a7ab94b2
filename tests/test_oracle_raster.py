"""Pins of the oracle's position-map rasteriser (the rendered position maps of
Sec. 3.1 from which the correspondence of Sec. 3.2 is built): closed-form
ray/plane positions, exact coverage of axis-aligned rectangles, occlusion,
near-plane culling, and agreement with the input module's independent
binary64 rasteriser on a curved mesh."""
import numpy as np

import oracle
from paper_2608_13255_gb300 import synth


def _world(cam, Xc):
    """camera-space points [..., 3] -> world (binary64), x_w = R^T (x_c - t)"""
    R = cam[:9].astype(np.float64).reshape(3, 3)
    t = cam[9:12].astype(np.float64)
    return (np.asarray(Xc, np.float64) - t) @ R


def _rect(cam, x0, x1, y0, y1, z):
    """two faces of a camera-space rectangle [x0,x1] x [y0,y1] at depth z"""
    V = _world(cam, [[x0, y0, z], [x1, y0, z], [x1, y1, z], [x0, y1, z]]).astype(np.float32)
    F = np.array([[0, 1, 2], [0, 2, 3]], np.int32)
    return V, F


def _rays(cam, H, W):
    fx, fy, cx, cy = (float(v) for v in cam[12:16])
    jj, ii = np.meshgrid(np.arange(H) + 0.5, np.arange(W) + 0.5, indexing="ij")
    return np.stack([(ii - cx) / fx, (jj - cy) / fy, np.ones_like(ii)], -1)  # camera-space directions


def test_quad_filling_the_view_gives_ray_plane_positions():
    H, W = 24, 40
    cam = synth.look_at_camera(30.0, 20.0, H, W)
    V, F = _rect(cam, -20.0, 20.0, -20.0, 20.0, 3.0)
    pos, valid = oracle.raster(V, F, cam, H, W)
    assert valid.all()
    # the plane through the (float32) corners, intersected in binary64
    Vc = (V.astype(np.float64) @ cam[:9].astype(np.float64).reshape(3, 3).T) + cam[9:12].astype(np.float64)
    n = np.cross(Vc[1] - Vc[0], Vc[2] - Vc[0])
    d = _rays(cam, H, W)
    s = (n @ Vc[0]) / (d @ n)
    exact = _world(cam, d * s[..., None])
    np.testing.assert_allclose(pos, exact, atol=2e-5, rtol=0)


def test_rectangle_coverage_is_exact():
    H, W = 32, 32
    cam = synth.look_at_camera(0.0, 0.0, H, W)
    fx, cx = float(cam[12]), float(cam[14])
    z = 2.5
    # edges at projected u = 7.3 .. 21.8, v = 4.6 .. 27.1 (never on a pixel centre)
    x0, x1 = (7.3 - cx) * z / fx, (21.8 - cx) * z / fx
    y0, y1 = (4.6 - cx) * z / fx, (27.1 - cx) * z / fx
    V, F = _rect(cam, x0, x1, y0, y1, z)
    _, valid = oracle.raster(V, F, cam, H, W)
    ii = np.arange(W) + 0.5
    jj = np.arange(H) + 0.5
    expect = ((jj[:, None] > 4.6) & (jj[:, None] < 27.1) & (ii[None, :] > 7.3) & (ii[None, :] < 21.8))
    np.testing.assert_array_equal(valid > 0, expect)


def test_nearest_face_wins_in_any_order():
    H, W = 32, 32
    cam = synth.look_at_camera(45.0, 10.0, H, W)
    Vb, Fb = _rect(cam, -3.0, 3.0, -3.0, 3.0, 4.0)      # behind, fills the view
    Vf, Ff = _rect(cam, -0.5, 0.7, -0.6, 0.4, 2.0)      # in front, a smaller patch
    for order in (0, 1):
        parts = [(Vb, Fb), (Vf, Ff)] if order == 0 else [(Vf, Ff), (Vb, Fb)]
        V = np.concatenate([parts[0][0], parts[1][0]])
        F = np.concatenate([parts[0][1], parts[1][1] + len(parts[0][0])])
        pos, valid = oracle.raster(V, F, cam, H, W)
        assert valid.all()
        depth = ((pos.astype(np.float64) @ cam[:9].astype(np.float64).reshape(3, 3).T)
                 + cam[9:12].astype(np.float64))[..., 2]
        _, vf = oracle.raster(Vf, Ff, cam, H, W)
        np.testing.assert_allclose(depth[vf > 0], 2.0, atol=1e-5)
        np.testing.assert_allclose(depth[vf == 0], 4.0, atol=1e-5)
        assert 0 < (vf > 0).sum() < H * W


def test_faces_behind_the_camera_or_with_bad_indices_are_skipped():
    H, W = 16, 16
    cam = synth.look_at_camera(0.0, 0.0, H, W)
    V = _world(cam, [[-1.0, -1.0, 2.0], [1.0, -1.0, 2.0], [0.0, 1.0, -0.5]]).astype(np.float32)
    _, valid = oracle.raster(V, np.array([[0, 1, 2]], np.int32), cam, H, W)
    assert not valid.any()
    V2, F2 = _rect(cam, -5.0, 5.0, -5.0, 5.0, 3.0)
    _, valid = oracle.raster(V2, np.array([[0, 1, 7], [0, 2, 3]], np.int32), cam, H, W)
    assert 0 < valid.sum() < H * W  # only the second face remains


def test_agrees_with_the_input_modules_binary64_rasteriser():
    rng = np.random.default_rng(4)
    V, F = synth.blob_mesh(3, 0.15, rng)
    H = W = 64
    for az, el in synth.hunyuan_layout():
        cam = synth.look_at_camera(az, el, H, W)
        p32, v32 = oracle.raster(V.astype(np.float32), F, cam, H, W)
        p64, v64 = synth.raster_mesh(V, F, cam, H, W)
        assert (v32 != v64).mean() < 2e-3  # silhouette pixels decided within rounding
        both = (v32 > 0) & (v64 > 0)
        assert both.sum() > 0.2 * H * W
        err = np.abs(p32[both] - p64[both]).max(-1)
        assert np.quantile(err, 0.999) < 1e-4
