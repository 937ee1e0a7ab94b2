"""GPU parity: the CUDA path, called through the C ABI, against the CPU oracle
on identical seeded inputs (Sec. 3.2: correspondence operator, Eq. 1 delta
transport with multi-anchor aggregation, sampler reconstruction, full-step
passthrough).  Indices must match bit for bit (target pixels inside the
threshold band are counted and excluded); latents must meet the tolerances
stated in gpu_helpers."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_13255_gb300 import synth

from gpu_helpers import (DeviceGeometry, assert_bf16_close, assert_f32_close, latent_values, lat_torch_dtype,
                         pred_scale, recon_kw, step_inputs)

pytestmark = pytest.mark.gpu

WORKLOADS = ["tiny", "hunyuan64", "solids96", "ring12_128", "batch128"]


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13255_gb300 import build as gbuild
    gbuild.build()
    from paper_2608_13255_gb300 import geocache
    geocache.load()
    return geocache


def _compare_tables(w, g, K):
    tau_ref = oracle.tau(w.pos, w.valid, w.tol_frac)
    np.testing.assert_array_equal(g.tau.cpu().numpy(), tau_ref)  # bit-exact tau
    idx_ref, w_ref, band = oracle.build_corr(w.pos, w.valid, w.cams, tau_ref, K=K)
    idx = g.idx.cpu().numpy()
    wt = g.wt.cpu().numpy()
    inband = np.broadcast_to(band[..., None] > 0, idx.shape)
    mism = (idx != idx_ref) & ~inband
    assert not mism.any(), "%d index mismatches outside the threshold band" % mism.sum()
    kept = idx_ref >= 0
    assert_f32_close(wt[~inband], w_ref[~inband], what="weights")
    # keep masks: bit k set iff tap k is kept
    keep_ref = sum((kept[..., k].astype(np.uint8) << k) for k in range(K))
    keep = g.keep.cpu().numpy()
    assert not ((keep != keep_ref) & (band == 0)).any(), "keep masks differ outside the threshold band"
    # sparse form: one record per kept row, in (b, v, u, token) order, whose
    # taps are the table's taps
    if not band.any():
        rec = g.records.cpu().numpy()[: g.n_records]
        tp = g.tile_ptr.cpu().numpy()
        T = g.gc.tiles_per_view(w.H, w.W)
        rows = np.flatnonzero(keep_ref.reshape(-1) > 0)  # (b, v, u, p) order
        assert g.n_records == len(rows) == tp[-1]
        HW = w.H * w.W
        p = rows % HW
        assert (rec[:, 0] & 0x0FFFFFFF == p).all()
        assert ((rec[:, 0] >> 28) & 15 == keep_ref.reshape(-1)[rows]).all()
        pair = rows // HW
        counts = np.bincount(pair * T + p // 1024, minlength=w.B * w.N * w.N * T)
        np.testing.assert_array_equal(tp, np.concatenate([[0], np.cumsum(counts)]))
        q_tl = rec[:, 1].astype(np.int64)
        ir = idx_ref.reshape(-1, K)[rows]
        offs = np.array([0, 1, w.W, w.W + 1])[:K] if K == 4 else np.array([0])
        expect = np.where(ir >= 0, q_tl[:, None] + offs[None, :], -1)
        np.testing.assert_array_equal(expect, ir)
    return int(band.sum()), float(kept.any(-1).mean())


@pytest.mark.parametrize("name", WORKLOADS)
def test_tables_bit_exact(gc, workloads, name):
    w = workloads(name)
    g = DeviceGeometry(w, K=w.K)
    torch.cuda.synchronize()
    nband, cover = _compare_tables(w, g, w.K)
    print("%s: threshold-band pixels %d, rows with a kept tap %.4f" % (name, nband, cover))


@pytest.mark.parametrize("name", ["tiny", "solids96"])
def test_tables_bit_exact_k1(gc, workloads, name):
    w = workloads(name)
    g = DeviceGeometry(w, K=1)
    torch.cuda.synchronize()
    _compare_tables(w, g, 1)


def _run_step(gc, w, g, anchors, params, pred=None, mode="sparse", inplace=False, xinplace=False,
              seed_extra=0, C=None, minimal_ws=False):
    """One cached step on the GPU and in the oracle from the same inputs."""
    if C is not None and C != w.C:
        w = synth.Workload(**{**w.__dict__, "C": C})
    x0_prev, x0_new, xt32 = step_inputs(w, 3, anchors, seed_extra)
    xt64, xt_t = latent_values(xt32, w)
    dev = "cuda"
    d_prev = torch.from_numpy(x0_prev).to(dev)
    d_new = torch.from_numpy(x0_new).to(dev)
    d_out = d_prev if inplace else torch.empty_like(d_prev)
    d_xt = xt_t.to(dev)
    d_xn = d_xt if xinplace else torch.empty_like(d_xt)
    d_pred = torch.empty_like(d_prev) if pred else None
    corr = g.corr_for(mode)
    r = gc.make_recon(params["sampler"], a_t=params.get("a_t", 0), a_prev=params.get("a_prev", 0),
                      sigma=params.get("sigma", 0), sigma_next=params.get("sigma_next", 0),
                      pred_kind=pred, pred_out=d_pred)
    gc.transport_step(corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r,
                      workspace=g.workspace(w.C, minimal=minimal_ws))
    torch.cuda.synchronize()
    gc.device_status()
    tau_ref = oracle.tau(w.pos, w.valid, w.tol_frac)
    ref_x0, ref_xn, ref_pred = oracle.transport_step(
        anchors, x0_new, x0_prev, K=g.corr.c.K, geom=(w.pos, w.valid, w.cams, tau_ref), x_t=xt64,
        recon=recon_kw(params, pred))
    got_x0 = d_out.cpu().numpy()
    e0 = assert_f32_close(got_x0, ref_x0, what="x0")
    if w.dtype == "bf16":
        bits = d_xn.cpu().view(torch.int16).numpy().view(np.uint16)
        e1 = assert_bf16_close(bits, ref_xn, what="x_next")[0]
    else:
        e1 = assert_f32_close(d_xn.cpu().numpy(), ref_xn, scale=2.0, what="x_next")
    if pred:
        assert_f32_close(d_pred.cpu().numpy(), ref_pred, scale=pred_scale(params), what="pred")
    return e0, e1, got_x0, ref_x0


def _first_cached(w):
    sched = w.schedule
    for t in range(w.S + 1):
        if not oracle.is_full_step(t, max(w.S, 2), sched):
            return t
    raise AssertionError


@pytest.mark.parametrize("name", WORKLOADS)
def test_transport_step_parity(gc, workloads, name):
    w = workloads(name)
    g = DeviceGeometry(w, K=w.K)
    t = _first_cached(w)
    anchors = oracle.rotate_anchors(w.N, w.a, oracle.cached_ordinal(t, max(w.S, 2), w.schedule))
    params = synth.recon_params(w, min(t, w.S - 1))
    e0, e1, got, ref = _run_step(gc, w, g, anchors, params)
    # the increment is really transported somewhere (non-trivial check)
    x0_prev = step_inputs(w, 3, anchors)[0]
    non = [v for v in range(w.N) if v not in anchors]
    moved = np.abs(ref[:, non] - x0_prev[:, non]).max()
    assert moved > 1e-3
    print("%s anchors %s: max |dx0| %.3g, max |dx_next| %.3g" % (name, anchors, e0, e1))


@pytest.mark.parametrize("name,K", [("hunyuan64", 4), ("ring12_128", 4), ("solids96", 1)])
def test_corr_modes_agree_bitwise(gc, workloads, name, K):
    # sparse records, keep masks, full geometry and tables give the same
    # taps, weights and results
    w = workloads(name)
    g = DeviceGeometry(w, K=K)
    anchors = oracle.rotate_anchors(w.N, w.a, 1)
    params = synth.recon_params(w, 7)
    _, _, got_sparse, _ = _run_step(gc, w, g, anchors, params, mode="sparse")
    _, _, got_mask, _ = _run_step(gc, w, g, anchors, params, mode="mask")
    np.testing.assert_array_equal(got_sparse, got_mask)
    _, _, got_geom, _ = _run_step(gc, w, g, anchors, params, mode="geometry")
    _, _, got_tab, _ = _run_step(gc, w, g, anchors, params, mode="table")
    np.testing.assert_array_equal(got_mask, got_geom)
    np.testing.assert_array_equal(got_mask, got_tab)


@pytest.mark.parametrize("pred", ["eps", "v"])
def test_ddim_prediction_outputs(gc, workloads, pred):
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    for step in (1, 13, 28):
        params = synth.recon_params(w, step)
        _run_step(gc, w, g, [0, 3], params, pred=pred)


def test_fm_velocity_and_k1(gc, workloads):
    w = workloads("solids96")
    g = DeviceGeometry(w, K=1, tables=False)
    for step in (1, 25, 49):
        _run_step(gc, w, g, [1, 3, 5], synth.recon_params(w, step), pred="velocity")


@pytest.mark.parametrize("name,K,C,inplace", [("solids96", 1, 12, False), ("tiny", 4, 9, False),
                                               ("tiny", 1, 16, True)])
def test_plane_path_k1_and_f32(gc, workloads, name, K, C, inplace):
    # the increment-plane path (C >= 8) with one tap per record and with f32
    # latents: equal to the oracle, and bitwise to the record-parallel apply
    w = workloads(name)
    g = DeviceGeometry(w, K=K, tables=False, source_index=False)
    anchors = [1, 3, 5] if w.N == 6 and w.a == 3 else [0, 3]
    params = synth.recon_params(w, 1 if w.S > 1 else 0)
    _, _, got_plane, _ = _run_step(gc, w, g, anchors, params, C=C, inplace=inplace)
    _, _, got_rows, _ = _run_step(gc, w, g, anchors, params, C=C, inplace=inplace, minimal_ws=True)
    np.testing.assert_array_equal(got_plane, got_rows)


def test_in_place_cache_and_latents(gc, workloads):
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    params = synth.recon_params(w, 4)
    _, _, a, _ = _run_step(gc, w, g, [1, 4], params)
    for mode in ("sparse", "mask"):
        _, _, b, _ = _run_step(gc, w, g, [1, 4], params, inplace=True, xinplace=True, mode=mode)
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("C", [1, 3, 5, 16, 20, 33])
def test_channel_counts(gc, workloads, C):
    w = workloads("solids96")
    g = DeviceGeometry(w, K=4, tables=False)
    _run_step(gc, w, g, [0, 2, 4], synth.recon_params(w, 9), C=C)


@pytest.mark.parametrize("a", [1, 5])
def test_anchor_counts(gc, workloads, a):
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    _run_step(gc, w, g, oracle.rotate_anchors(w.N, a, 2), synth.recon_params(w, 2))


def test_ragged_tiles_and_many_views(gc):
    # 37x53 tokens (not a multiple of the 256-token tile), 3 assets, 6 views
    w = synth.make_workload("batch128", B=3, H=37, W=53)
    w9 = synth.Workload(**{**w.__dict__, "N": 6})
    g = DeviceGeometry(w9, K=4)
    torch.cuda.synchronize()
    _compare_tables(w9, g, 4)
    _run_step(gc, w9, g, [2, 5], synth.recon_params(w9, 11))
    # 64 views (the ABI maximum) on an 8x8 grid
    wv = synth.make_workload("tiny", H=8, W=8)
    cams = np.stack([synth.look_at_camera(360.0 * i / 64, 15.0 * ((i % 5) - 2), 8, 8) for i in range(64)])[None]
    pos, valid = synth.render_asset(synth.unit_sphere(), cams[0], 8, 8)
    wv = synth.Workload(**{**wv.__dict__, "N": 64, "cams": cams.astype(np.float32), "pos": pos[None],
                           "valid": valid[None]})
    g = DeviceGeometry(wv, K=4)
    torch.cuda.synchronize()
    _compare_tables(wv, g, 4)
    _run_step(gc, wv, g, oracle.rotate_anchors(64, 8, 3), synth.recon_params(wv, 0))
    # more anchors than the tiled kernel holds (general per-token kernel), K = 4 and K = 1
    _run_step(gc, wv, g, oracle.rotate_anchors(64, 12, 1), synth.recon_params(wv, 0))
    _run_step(gc, wv, g, oracle.rotate_anchors(64, 12, 1), synth.recon_params(wv, 0), mode="table")


@pytest.mark.parametrize("seed", range(6))
def test_random_shapes_split_the_grid_right(gc, seed):
    # random (B, N, a, C, H, W): the step kernels split their block index into
    # (asset, view, tile, channel group, record slice) with launch-invariant
    # divisors; every shape must still equal the oracle, and the sparse step
    # the mask-mode step bit for bit (both with and without the increment plane)
    rng = np.random.default_rng(9000 + seed)
    B, N = int(rng.integers(1, 4)), int(rng.integers(2, 11))
    a, C = int(rng.integers(1, N)), int(rng.integers(1, 21))
    H, W = int(rng.integers(7, 76)), int(rng.integers(7, 76))
    cams = np.stack([synth.look_at_camera(az + 11.0 * seed, el, H, W)
                     for az, el in synth.ring_layout(N, el_deg=10.0)]).astype(np.float32)
    shapes = [synth.unit_sphere() if b % 2 == 0 else synth.random_solids(np.random.default_rng(seed * 10 + b))
              for b in range(B)]
    maps = [synth.render_asset(sh, cams, H, W) for sh in shapes]
    w = synth.make_workload("tiny", H=H, W=W)
    w = synth.Workload(**{**w.__dict__, "B": B, "N": N, "a": a, "C": C, "dtype": "bf16", "sampler": "ddim", "S": 30,
                          "cams": np.ascontiguousarray(np.tile(cams[None], (B, 1, 1))),
                          "pos": np.stack([m[0] for m in maps]), "valid": np.stack([m[1] for m in maps])})
    g = DeviceGeometry(w, K=4, tables=False, source_index=False)
    anchors = sorted(rng.choice(N, size=a, replace=False).tolist())
    params = synth.recon_params(w, 7)
    _, _, got_sparse, _ = _run_step(gc, w, g, anchors, params)
    _, _, got_min, _ = _run_step(gc, w, g, anchors, params, minimal_ws=True)
    _, _, got_mask, _ = _run_step(gc, w, g, anchors, params, mode="mask")
    np.testing.assert_array_equal(got_sparse, got_mask)
    np.testing.assert_array_equal(got_min, got_mask)
    print("B=%d N=%d a=%d C=%d %dx%d anchors %s: %d records" % (B, N, a, C, H, W, anchors, g.n_records))


def test_empty_asset_keeps_state(gc, workloads):
    # an asset with no foreground: tau = 0, no taps, every target keeps x0
    w = workloads("hunyuan64")
    we = synth.Workload(**{**w.__dict__, "valid": np.zeros_like(w.valid), "pos": np.zeros_like(w.pos)})
    g = DeviceGeometry(we, K=4)
    torch.cuda.synchronize()
    assert g.tau.item() == 0.0
    assert (g.idx.cpu().numpy() == -1).all()
    _, _, got, _ = _run_step(gc, we, g, [0, 3], synth.recon_params(we, 1))
    x0_prev, x0_new, _ = step_inputs(we, 3, [0, 3])
    non = [1, 2, 4, 5]
    np.testing.assert_array_equal(got[:, non], x0_prev[:, non])


def test_zero_delta_bit_identical(gc, workloads):
    w = workloads("ring12_128")
    g = DeviceGeometry(w, K=4, tables=False)
    x0_prev, _, _ = step_inputs(w, 3, [0, 3, 6, 9])  # keep-mask path
    d_prev = torch.from_numpy(x0_prev).cuda()
    d_new = d_prev[:, [0, 3, 6, 9]].contiguous()
    d_out = torch.empty_like(d_prev)
    gc.transport_step(g.corr, [0, 3, 6, 9], w.C, d_new, d_prev, d_out, workspace=g.workspace(w.C))
    torch.cuda.synchronize()
    assert torch.equal(d_out, d_prev)


def test_all_anchor_step_equals_full_step(gc, workloads):
    # a = N: the cached step must equal the stock sampler step bit for bit
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    x0_prev, x0_new, xt32 = step_inputs(w, 3, list(range(w.N)))
    _, xt = latent_values(xt32, w)
    xt = xt.cuda()
    p = synth.recon_params(w, 12)
    r = gc.make_recon("ddim", a_t=p["a_t"], a_prev=p["a_prev"])
    d_new = torch.from_numpy(x0_new).cuda()
    out1, xn1 = torch.empty_like(d_new), torch.empty_like(xt)
    gc.transport_step(g.corr, list(range(w.N)), w.C, d_new, torch.from_numpy(x0_prev).cuda(), out1, xt, xn1, r,
                      workspace=g.workspace(w.C))
    xn2 = torch.empty_like(xt)
    gc.reconstruct(xt, d_new, xn2, r)
    torch.cuda.synchronize()
    assert torch.equal(out1, d_new)
    assert torch.equal(xn1.view(torch.int16), xn2.view(torch.int16))


@pytest.mark.parametrize("name,pred", [("tiny", "eps"), ("hunyuan64", "v"), ("solids96", "velocity")])
def test_full_step_reconstruct_parity(gc, workloads, name, pred):
    w = workloads(name)
    rng = np.random.default_rng(11)
    x0 = rng.standard_normal((w.B, w.N, w.C, w.H, w.W), dtype=np.float32)
    xt64, xt = latent_values(rng.standard_normal(x0.shape, dtype=np.float32), w)
    step = 0 if name == "tiny" else 5
    p = synth.recon_params(w, step)
    d_pred = torch.empty(x0.shape, dtype=torch.float32, device="cuda")
    d_store = torch.empty_like(d_pred)
    r = gc.make_recon(p["sampler"], a_t=p.get("a_t", 0), a_prev=p.get("a_prev", 0), sigma=p.get("sigma", 0),
                      sigma_next=p.get("sigma_next", 0), pred_kind=pred, pred_out=d_pred)
    xt = xt.cuda()
    xn = torch.empty_like(xt)
    d_x0 = torch.from_numpy(x0).cuda()
    gc.reconstruct(xt, d_x0, xn, r, x0_store=d_store)
    torch.cuda.synchronize()
    ref_xn, ref_pred = oracle.reconstruct(xt64, x0.astype(np.float64), **recon_kw(p, pred))
    if w.dtype == "bf16":
        assert_bf16_close(xn.cpu().view(torch.int16).numpy().view(np.uint16), ref_xn, what="x_next")
    else:
        assert_f32_close(xn.cpu().numpy(), ref_xn, scale=2.0, what="x_next")
    assert_f32_close(d_pred.cpu().numpy(), ref_pred, scale=pred_scale(p), what="pred")
    assert torch.equal(d_store, d_x0)


def test_trajectory_per_step_parity_and_drift(gc, workloads):
    """Whole 30-step DDIM trajectory (full every 5, rotating anchors): each
    step is checked against the oracle from the GPU's own state; the drift
    of the GPU trajectory against the oracle's own binary64 trajectory is
    reported."""
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    ws = g.workspace(w.C)
    xT, x0_init = synth.initial_latents(w)
    tau_ref = oracle.tau(w.pos, w.valid)
    geom = (w.pos, w.valid, w.cams, tau_ref)
    xbits = synth.to_bf16_bits(xT)
    x = torch.from_numpy(xbits.view(np.int16)).view(torch.bfloat16).cuda()
    x_or = (xbits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)  # oracle's own state
    cache = None          # GPU x0 state
    cache_or = x0_init.astype(np.float64)  # oracle's own x0 state
    x0_prev_np = x0_init.copy()
    for t in range(w.S):
        p = synth.recon_params(w, t)
        r = gc.make_recon("ddim", a_t=p["a_t"], a_prev=p["a_prev"])
        rk = recon_kw(p)
        x_in64 = (x.cpu().view(torch.int16).numpy().view(np.uint16).astype(np.uint32) << 16
                  ).view(np.float32).astype(np.float64)
        if oracle.is_full_step(t, w.S, w.schedule):
            dl = synth.delta(w, t, list(range(w.N)))
            x0_full = (x0_prev_np + dl).astype(np.float32)
            d_full = torch.from_numpy(x0_full).cuda()
            xn = torch.empty_like(x)
            gc.reconstruct(x, d_full, xn, r)
            ref_xn, _ = oracle.reconstruct(x_in64, x0_full.astype(np.float64), **rk)
            cache = d_full
            cache_or = cache_or + dl
            x_or_next, _ = oracle.reconstruct(x_or, cache_or, **rk)
        else:
            anchors = oracle.rotate_anchors(w.N, w.a, oracle.cached_ordinal(t, w.S, w.schedule))
            dl = synth.delta(w, t, anchors)
            x0_new = (cache.cpu().numpy()[:, anchors] + dl).astype(np.float32)
            d_new = torch.from_numpy(x0_new).cuda()
            out = torch.empty_like(cache)
            xn = torch.empty_like(x)
            gc.transport_step(g.corr, anchors, w.C, d_new, cache, out, x, xn, r, workspace=ws)
            ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, cache.cpu().numpy(), geom=geom,
                                                      x_t=x_in64, recon=rk)
            torch.cuda.synchronize()
            assert_f32_close(out.cpu().numpy(), ref_x0, what="x0 step %d" % t)
            cache_or, x_or_next, _ = oracle.transport_step(anchors, cache_or[:, anchors] + dl, cache_or,
                                                           geom=geom, x_t=x_or, recon=rk)
            cache = out
        torch.cuda.synchronize()
        assert_bf16_close(xn.cpu().view(torch.int16).numpy().view(np.uint16), ref_xn, what="x step %d" % t)
        x = xn
        x0_prev_np = cache.cpu().numpy()
        x_or = (oracle.round_bf16(x_or_next).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    drift = np.abs(x.cpu().float().numpy().astype(np.float64) - x_or).max()
    print("end-of-trajectory drift (GPU vs oracle's own trajectory): %.4g" % drift)
    assert drift < 0.25


def test_record_overflow_is_reported_not_faulted(gc, workloads):
    # a sparse form built into too few records: the excess is dropped and
    # flagged in the device status word; a transport step over it reads only
    # the records that exist (no fault), and the status is reported
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    short = torch.empty((g.n_records // 2, 4), dtype=torch.int32, device="cuda")
    c = gc.make_corr(g.pos, g.valid, g.cams, g.tau, K=4, keep=g.keep, tile_ptr=g.tile_ptr, records=short,
                     mode=gc.CORR_SPARSE)
    gc.build_corr(c)
    with pytest.raises(gc.GeocacheError) as ei:
        gc.device_status()
    assert ei.value.status == gc.ESHAPE
    gc.device_status()  # cleared by the read
    x0_prev, x0_new, _ = step_inputs(w, 3, [0, 3])
    d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
    out = torch.empty_like(d_prev)
    ws = torch.empty(max(c.workspace_floats(w.C), 4), device="cuda")
    gc.transport_step(c, [0, 3], w.C, d_new, d_prev, out, workspace=ws)
    torch.cuda.synchronize()
    gc.device_status()
    assert torch.isfinite(out).all()


@pytest.mark.parametrize("name", ["hunyuan64", "ragged"])
def test_table_index_out_of_range_is_dropped_and_reported(gc, workloads, name):
    # a caller's correspondence table with indices outside the view (past the
    # last token, and below -1): a TABLE-mode step drops those taps instead of
    # reading outside the view, reports EINVAL through the device status word,
    # and equals bit for bit the step on the same table with those taps
    # removed (64 x 64: the staged kernel; 37 x 53: the per-tile kernel)
    w = workloads("hunyuan64") if name == "hunyuan64" else synth.make_workload("batch128", B=1, H=37, W=53)
    g = DeviceGeometry(w, K=4, tables=True)
    torch.cuda.synchronize()
    HW = w.H * w.W
    idx, wt = g.idx.clone(), g.wt.clone()
    kept = torch.nonzero(idx.view(-1) >= 0).view(-1)
    bad = kept[torch.randperm(kept.numel(), generator=torch.Generator().manual_seed(4))[:64].cuda()]
    idx.view(-1)[bad[:32]] = HW + 5
    idx.view(-1)[bad[32:]] = -7
    clean_idx, clean_wt = idx.clone(), wt.clone()
    clean_idx.view(-1)[bad] = -1
    clean_wt.view(-1)[bad] = 0.0
    anchors = [0, 3]
    x0_prev, x0_new, _ = step_inputs(w, 3, anchors)
    d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
    outs = []
    for ti, tw in ((idx, wt), (clean_idx, clean_wt)):
        c = gc.make_corr(g.pos, g.valid, g.cams, g.tau, ti, tw, K=4, tol_frac=w.tol_frac, mode=gc.CORR_TABLE)
        out = torch.empty_like(d_prev)
        gc.transport_step(c, anchors, w.C, d_new, d_prev, out)
        torch.cuda.synchronize()
        outs.append(out)
        if ti is idx:
            with pytest.raises(gc.GeocacheError) as ei:
                gc.device_status()
            assert ei.value.status == gc.EINVAL and "table index" in str(ei.value)
        gc.device_status()  # clean
    assert torch.isfinite(outs[0]).all()
    assert torch.equal(outs[0].view(torch.int32), outs[1].view(torch.int32))


def test_graph_replay_matches_eager(gc, workloads):
    # a cached step captured in a CUDA graph (with the programmatic
    # dependency between its two kernels) gives the eager results
    w = workloads("batch128")
    g = DeviceGeometry(w, K=4, tables=False)
    x0_prev, x0_new, xt32 = step_inputs(w, 5, [1, 4])
    _, xt = latent_values(xt32, w)
    d_prev, d_new, d_xt = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda(), xt.cuda()
    ws = g.workspace(w.C)
    p = synth.recon_params(w, 5)
    r = gc.make_recon("ddim", a_t=p["a_t"], a_prev=p["a_prev"])
    out_e, xn_e = torch.empty_like(d_prev), torch.empty_like(d_xt)
    gc.transport_step(g.corr, [1, 4], w.C, d_new, d_prev, out_e, d_xt, xn_e, r, workspace=ws)
    out_g, xn_g = torch.empty_like(d_prev), torch.empty_like(d_xt)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        gc.transport_step(g.corr, [1, 4], w.C, d_new, d_prev, out_g, d_xt, xn_g, r, workspace=ws)
    graph.replay()
    torch.cuda.synchronize()
    assert torch.equal(out_g, out_e)
    assert torch.equal(xn_g.view(torch.int16), xn_e.view(torch.int16))


@pytest.mark.parametrize("K", [4, 1])
@pytest.mark.parametrize("scene", ["plane", "asset"])
def test_identity_camera_reproduces_anchor_delta(gc, workloads, scene, K):
    """Target camera equal to the anchor camera (Sec. 3.2, correspondence
    operator): the taps sit on the target's own token, where floor(u - 0.5)
    and the zero-weight rule decide the tap set.  'plane': positions that
    project exactly onto the token centres (one tap, weight 1, for K = 4 as
    for K = 1); 'asset': a rendered view duplicated (projections within
    rounding of the centres).  Tables bit-exact against the oracle; x0^1(t) -
    x0^1(t-1) = delta^0 at every foreground token, bit for bit where the
    single tap has weight 1 and within 1e-5 otherwise; SPARSE, TABLE and MASK
    modes bitwise equal."""
    w = synth.identity_camera_pair(workloads("hunyuan64"), view=1, plane=(scene == "plane"))
    g = DeviceGeometry(w, K=K)
    torch.cuda.synchronize()
    nband, _ = _compare_tables(w, g, K)
    assert nband == 0
    fg = w.valid[0, 1].reshape(-1) > 0
    p = np.flatnonzero(fg)
    idx = g.idx.cpu().numpy()[0, 1, 0].reshape(-1, K)
    wt = g.wt.cpu().numpy()[0, 1, 0].reshape(-1, K)
    dominant = np.take_along_axis(idx[fg], wt[fg].argmax(1)[:, None], 1)[:, 0]
    np.testing.assert_array_equal(dominant, p)  # the heaviest tap is the target's own token
    exact = scene == "plane" or K == 1
    if exact:
        np.testing.assert_array_equal(idx[fg, 0], p)
        assert (wt[fg, 0] == 1.0).all() and (idx[fg, 1:] == -1).all()
    else:
        assert wt[fg].max(1).min() >= 1.0 - 1e-4
    anchors = [0]
    params = synth.recon_params(w, 9)
    outs = {}
    for mode in ("sparse", "table", "mask"):
        _, _, got, ref = _run_step(gc, w, g, anchors, params, mode=mode)
        outs[mode] = got
    np.testing.assert_array_equal(outs["sparse"], outs["table"])
    np.testing.assert_array_equal(outs["sparse"], outs["mask"])
    x0_prev, x0_new, _ = step_inputs(w, 3, anchors)
    got = outs["sparse"][0, 1].reshape(w.C, -1)
    prev = x0_prev[0, 1].reshape(w.C, -1)
    d0 = (x0_new[0, 0] - x0_prev[0, 0]).reshape(w.C, -1)  # binary32, as the kernel forms it
    np.testing.assert_array_equal(got[:, ~fg], prev[:, ~fg])  # background keeps its state
    if exact:  # one tap of weight 1: x0(t) = x0(t-1) + delta in binary32, bit for bit
        np.testing.assert_array_equal(got[:, fg], (prev + d0)[:, fg])
    err = np.abs((got.astype(np.float64) - prev)[:, fg] - d0[:, fg].astype(np.float64))
    assert err.max() <= 1e-5, err.max()
    print("%s K=%d: %d foreground tokens, max |x0(t) - x0(t-1) - delta| %.3g" % (scene, K, fg.sum(), err.max()))


def _source_groups(g, w):
    """Expected source index from the records: for every record r of pair
    (b, v, u), its group (b, u, tile of its first kept tap) and target v."""
    T = g.gc.tiles_per_view(w.H, w.W)
    rec = g.records.cpu().numpy()[: g.n_records].astype(np.int64)
    tp = g.tile_ptr.cpu().numpy().astype(np.int64)
    pair = np.repeat(np.arange(w.B * w.N * w.N), tp[T::T] - tp[:-1:T])  # (b, v, u) of each record
    b, v, u = pair // (w.N * w.N), (pair // w.N) % w.N, pair % w.N
    mask, q_tl = (rec[:, 0] >> 28) & 15, rec[:, 1]
    low = np.array([0, 0, 1, 0, 2, 0, 1, 0, 3, 0, 1, 0, 2, 0, 1, 0])[mask]  # lowest kept tap
    q = q_tl + (low & 1) + (low >> 1) * w.W if w.K == 4 else q_tl
    return (b * w.N + u) * T + q // 1024, v


@pytest.mark.parametrize("name", ["ring12_128", "solids96"])
def test_source_index_groups_every_record_once(gc, workloads, name):
    # the source index (records grouped by the tile of their first kept tap in
    # the source view) holds each record exactly once, in the right group,
    # with its target view
    w = workloads(name)
    g = DeviceGeometry(w, K=w.K, tables=False)
    torch.cuda.synchronize()
    grp, v = _source_groups(g, w)
    ends = g.src_ptr.cpu().numpy().astype(np.int64)
    starts = np.concatenate([[0], ends[:-2]])
    ent = g.src_rec.cpu().numpy()[: g.n_records]
    assert ends[-2] == ends[-1] == g.n_records
    np.testing.assert_array_equal(ends[:-1] - starts, np.bincount(grp, minlength=len(ends) - 1))
    got_grp = np.repeat(np.arange(len(ends) - 1), ends[:-1] - starts)
    order = np.argsort(ent[:, 0], kind="stable")
    np.testing.assert_array_equal(np.sort(ent[:, 0]), np.arange(g.n_records))  # every record once
    np.testing.assert_array_equal(got_grp[order], grp)
    np.testing.assert_array_equal(ent[order, 1], v)


@pytest.mark.parametrize("C,update,inplace", [(16, "delta", False), (16, "delta", True), (20, "copy", False),
                                              (33, "delta", False), (8, "copy", True)])
def test_wide_latent_paths_agree_bitwise(gc, workloads, C, update, inplace):
    # wide latents (C >= 8) have three ways to form the records' increments:
    # the anchors' increment plane (workspace with room for it), the
    # source-tile apply (minimal workspace, corr with a source index) and the
    # record-parallel apply (minimal workspace, no index).  All three give the
    # same bits, and the oracle's results.
    w = workloads("ring12_128") if C == 16 else workloads("solids96")
    w = synth.Workload(**{**w.__dict__, "C": C})
    g = DeviceGeometry(w, K=w.K, tables=False)
    anchors = oracle.rotate_anchors(w.N, w.a, 1)
    params = synth.recon_params(w, 8)
    outs = {}
    for path, mode, minimal in (("plane", "sparse_plain", False), ("source_tile", "sparse", True),
                                ("record", "sparse_plain", True)):
        ws = g.workspace(C, minimal=minimal)
        if not minimal:  # room for max_records * C floats and the plane
            assert ws.numel() >= g.corr.min_workspace_floats(C) + len(anchors) * w.B * -(-C // 4) * 4 * w.H * w.W
        x0_prev, x0_new, xt32 = step_inputs(w, 3, anchors)
        xt64, xt = latent_values(xt32, w)
        d_prev, d_new, d_xt = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda(), xt.cuda()
        d_out = d_prev if inplace else torch.empty_like(d_prev)
        d_xn = d_xt if inplace else torch.empty_like(d_xt)
        r = gc.make_recon(params["sampler"], a_t=params.get("a_t", 0), a_prev=params.get("a_prev", 0),
                          sigma=params.get("sigma", 0), sigma_next=params.get("sigma_next", 0))
        gc.transport_step(g.corr_for(mode), anchors, C, d_new, d_prev, d_out, d_xt, d_xn, r, workspace=ws,
                          update=update)
        torch.cuda.synchronize()
        gc.device_status()
        outs[path] = (d_out.cpu().numpy(), d_xn.cpu().view(torch.int16).numpy())
    for path in ("source_tile", "record"):
        np.testing.assert_array_equal(outs[path][0], outs["plane"][0])
        np.testing.assert_array_equal(outs[path][1], outs["plane"][1])
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=w.K, geom=(w.pos, w.valid, w.cams, tau),
                                              x_t=xt64, recon=recon_kw(params), update=update)
    assert_f32_close(outs["plane"][0], ref_x0, what="x0")
    assert_bf16_close(outs["plane"][1].view(np.uint16), ref_xn, what="x_next")


def test_wide_views_fall_back_to_the_record_parallel_apply(gc):
    # W + 1 > 1024 tokens: the staged span of a source tile would not fit, so a
    # step with a source index and a minimal workspace applies the records
    # record-parallel; with room for the increment plane (no span limit) it
    # takes the plane.  Both equal the oracle's results.
    H, W = 16, 1040
    w = synth.make_workload("solids96", H=H, W=W)
    cams = np.stack([synth.look_at_camera(az, el, W, W) for az, el in synth.hunyuan_layout()])
    cams[:, 15] = H / 2.0  # a 16-row strip through the middle of a square camera's image
    pos, valid = synth.render_asset(synth.unit_sphere(), cams, H, W)
    w = synth.Workload(**{**w.__dict__, "C": 8, "cams": cams[None].astype(np.float32), "pos": pos[None],
                          "valid": valid[None]})
    g = DeviceGeometry(w, K=4, tables=False)
    assert g.n_records > 100
    _, _, x0_min, _ = _run_step(gc, w, g, [0, 2, 4], synth.recon_params(w, 5), minimal_ws=True)
    _, _, x0_plane, _ = _run_step(gc, w, g, [0, 2, 4], synth.recon_params(w, 5))
    np.testing.assert_array_equal(x0_min, x0_plane)