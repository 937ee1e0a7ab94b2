"""GPU parity of the position-map rasteriser (geocache_raster_posmaps; the
rendered position maps of Sec. 3.1) against the oracle's binary32 z-buffer,
through the C ABI.  Both sides take every decision and form every position
in binary32 in the same order, so validity and positions must agree bit for
bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_13255_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13255_gb300 import build as gbuild
    gbuild.build()
    from paper_2608_13255_gb300 import geocache
    geocache.load()
    return geocache


def _big_quads(cam):
    """a view-filling rectangle behind a smaller one (faces far larger than a warp's box)"""
    R = cam[:9].astype(np.float64).reshape(3, 3)
    t = cam[9:12].astype(np.float64)
    pts = []
    for (x0, x1, y0, y1, z) in ((-3.0, 3.0, -3.0, 3.0, 4.0), (-0.6, 0.5, -0.4, 0.7, 2.0)):
        pts += [[x0, y0, z], [x1, y0, z], [x1, y1, z], [x0, y1, z]]
    V = ((np.array(pts) - t) @ R).astype(np.float32)
    F = np.array([[0, 1, 2], [0, 2, 3], [4, 5, 6], [4, 6, 7]], np.int32)
    return V, F


def _batch(H, W, N_layout):
    rng = np.random.default_rng(21)
    cams = np.stack([np.stack([synth.look_at_camera(az, el, H, W) for az, el in N_layout])] * 4)
    meshes = [synth.blob_mesh(4, 0.15, rng), synth.torus_mesh(), _big_quads(cams[2, 0]),
              (np.zeros((0, 3), np.float32), np.zeros((0, 3), np.int32))]
    meshes = [(np.asarray(V, np.float32), np.asarray(F, np.int32)) for V, F in meshes]
    return meshes, cams


def _upload(meshes, cams):
    v_off = np.cumsum([0] + [len(V) for V, _ in meshes])
    f_off = np.cumsum([0] + [len(F) for _, F in meshes]).astype(np.int64)
    verts = np.concatenate([V for V, _ in meshes]).astype(np.float32)
    faces = np.concatenate([F + v_off[b] for b, (_, F) in enumerate(meshes)]).astype(np.int32)
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
    return d(verts), d(faces), d(f_off), d(cams)


@pytest.mark.parametrize("H,W", [(64, 64), (48, 80)])
def test_posmaps_bit_exact(gc, H, W):
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    verts, faces, f_off, d_cams = _upload(meshes, cams)
    pos, valid = gc.raster_posmaps(verts, faces, f_off, d_cams, H, W)
    torch.cuda.synchronize()
    gc.device_status()
    pos, valid = pos.cpu().numpy(), valid.cpu().numpy()
    for b, (V, F) in enumerate(meshes):
        ref_p, ref_v = oracle.raster_views(V, F, cams[b], H, W)
        np.testing.assert_array_equal(valid[b], ref_v)
        np.testing.assert_array_equal(pos[b].view(np.uint32), ref_p.view(np.uint32))
    assert valid[0].mean() > 0.1 and valid[1].mean() > 0.05 and valid[2, 0].all() and not valid[3].any()


def test_posmaps_feed_the_correspondence_build(gc):
    # the rasterised maps of a blob are a valid input of the correspondence
    # build, which then gives the oracle's tables
    H = W = 64
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    verts, faces, f_off, d_cams = _upload(meshes[:1], cams[:1])
    pos, valid = gc.raster_posmaps(verts, faces, f_off, d_cams, H, W)
    tau = torch.zeros(1, dtype=torch.float32, device="cuda")
    keep = torch.empty((1, 6, 6, H, W), dtype=torch.uint8, device="cuda")
    c = gc.make_corr(pos, valid, d_cams, tau, keep=keep, mode=gc.CORR_MASK)
    gc.build_corr(c)
    ref_p, ref_v = oracle.raster_views(*meshes[0], cams[0], H, W)
    tau_ref = oracle.tau(ref_p[None], ref_v[None])
    np.testing.assert_array_equal(tau.cpu().numpy(), tau_ref)
    idx, _, band = oracle.build_corr(ref_p[None], ref_v[None], cams[:1], tau_ref, K=4)
    keep_ref = sum(((idx[..., k] >= 0).astype(np.uint8) << k) for k in range(4))
    assert not ((keep.cpu().numpy() != keep_ref) & (band == 0)).any()
    assert (keep_ref > 0).mean() > 0.01


def test_bad_face_index_is_skipped_and_reported(gc):
    H = W = 32
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    V, F = meshes[0]
    F = F.copy()
    F[5, 1] = len(V) + 3
    verts, faces, f_off, d_cams = _upload([(V, F)], cams[:1])
    pos, valid = gc.raster_posmaps(verts, faces, f_off, d_cams, H, W)
    torch.cuda.synchronize()
    with pytest.raises(gc.GeocacheError) as ei:
        gc.device_status()
    assert ei.value.status == gc.EINVAL
    gc.device_status()
    ref_p, ref_v = oracle.raster_views(V, F, cams[0], H, W)
    np.testing.assert_array_equal(valid.cpu().numpy()[0], ref_v)
    np.testing.assert_array_equal(pos.cpu().numpy()[0].view(np.uint32), ref_p.view(np.uint32))


@pytest.mark.parametrize("s,H,W", [(2, 64, 64), (4, 32, 32), (8, 16, 16), (3, 24, 40)])
def test_supersampled_posmaps_bit_exact(gc, s, H, W):
    # rendered at s x the token grid and pooled to it (image-resolution maps
    # of Sec. 3.1 brought to the token grid of Sec. 3.2): validity and
    # positions equal the oracle's render at s x with pooling, bit for bit
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    verts, faces, f_off, d_cams = _upload(meshes, cams)
    pos, valid = gc.raster_posmaps(verts, faces, f_off, d_cams, H, W, s=s)
    torch.cuda.synchronize()
    gc.device_status()
    pos, valid = pos.cpu().numpy(), valid.cpu().numpy()
    for b, (V, F) in enumerate(meshes):
        ref_p, ref_v = oracle.raster_supersampled(V, F, cams[b], H, W, s)
        np.testing.assert_array_equal(valid[b], ref_v)
        np.testing.assert_array_equal(pos[b].view(np.uint32), ref_p.view(np.uint32))
    assert valid[0].mean() > 0.1 and valid[2, 0].all() and not valid[3].any()


def test_supersampling_factor_one_is_the_plain_render(gc):
    H, W = 48, 80
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    verts, faces, f_off, d_cams = _upload(meshes, cams)
    p1, v1 = gc.raster_posmaps(verts, faces, f_off, d_cams, H, W)
    zb = torch.empty((4, 6, H, W), dtype=torch.int64, device="cuda")
    p2 = torch.empty_like(p1)
    v2 = torch.empty_like(v1)
    gc.load().geocache_raster_posmaps_supersampled(
        verts.data_ptr(), verts.shape[0], faces.data_ptr(), faces.shape[0], f_off.data_ptr(), 4, d_cams.data_ptr(), 6,
        H, W, 1, zb.data_ptr(), p2.data_ptr(), v2.data_ptr(), None)
    torch.cuda.synchronize()
    assert torch.equal(v1, v2) and torch.equal(p1.view(torch.int32), p2.view(torch.int32))


@pytest.mark.parametrize("s,H,W", [(8, 32, 32), (3, 37, 53), (1, 16, 24)])
def test_pool_posmaps_bit_exact(gc, s, H, W):
    # caller-rendered fine maps pooled on the GPU: equal to the oracle's
    # pooling bit for bit (maps rendered by the oracle at s x, several views)
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    fine_p, fine_v = oracle.raster_views(*meshes[0], oracle.scaled_camera(cams[0], s), H * s, W * s)
    ref_p, ref_v = oracle.pool(fine_p, fine_v, s)
    pos, valid = gc.pool_posmaps(torch.from_numpy(fine_p).cuda(), torch.from_numpy(fine_v).cuda(), s)
    torch.cuda.synchronize()
    gc.device_status()
    np.testing.assert_array_equal(valid.cpu().numpy(), ref_v)
    np.testing.assert_array_equal(pos.cpu().numpy().view(np.uint32), ref_p.view(np.uint32))
    assert ref_v.mean() > 0.05


def test_supersampled_posmaps_feed_the_correspondence_build(gc):
    # pooled maps (s = 4) into geocache_build_corr: tau, keep masks, tables
    # and records bit-exact against the oracle built on the oracle's pooled maps
    H = W = 64
    s = 4
    meshes, cams = _batch(H, W, synth.hunyuan_layout())
    verts, faces, f_off, d_cams = _upload(meshes[:1], cams[:1])
    pos, valid = gc.raster_posmaps(verts, faces, f_off, d_cams, H, W, s=s)
    ref_p, ref_v = oracle.raster_supersampled(*meshes[0], cams[0], H, W, s)
    np.testing.assert_array_equal(valid.cpu().numpy()[0], ref_v)
    corr = gc.build_sparse_corr(pos, valid, d_cams, K=4, tables=True)
    torch.cuda.synchronize()
    gc.device_status()
    tau_ref = oracle.tau(ref_p[None], ref_v[None])
    np.testing.assert_array_equal(corr.tau.cpu().numpy(), tau_ref)
    idx, w, band = oracle.build_corr(ref_p[None], ref_v[None], cams[:1], tau_ref, K=4)
    inband = np.broadcast_to(band[..., None] > 0, idx.shape)
    assert not ((corr.idx.cpu().numpy() != idx) & ~inband).any()
    assert (idx >= 0).any(-1).mean() > 0.01


def test_supersampled_sizes_are_checked(gc):
    meshes, cams = _batch(16, 16, synth.hunyuan_layout())
    verts, faces, f_off, d_cams = _upload(meshes[:1], cams[:1])
    with pytest.raises(gc.GeocacheError) as ei:
        gc.raster_posmaps(verts, faces, f_off, d_cams, 16, 16, s=17)
    assert ei.value.status == gc.ESHAPE
