"""Benchmark of the geometric delta transport on GB300.

One bench step = one pass of the whole hot path over a batch of assets:
tau (per-asset tolerance), then a DDIM trajectory of S sampler steps in which
the host picks full / cached and the rotating anchors, cached steps run the
fused correspondence + delta transport + reconstruction kernel, and full
steps run the passthrough reconstruction.  The denoiser's x0 outputs are
seeded synthetic tensors already resident in HBM.

value = target view-pixels transported + reconstructed per second, i.e.
sum over cached steps of B * (N - a) * H * W, divided by the trajectory time.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun each rank runs its own batch of assets (weak scaling, no
collective on the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "target view-pixels transported+reconstructed/sec per step; % of GB300 HBM BW"
UNIT = "target view-pixels/s"
L2_BYTES = 129 * 1024 * 1024


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=500)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="batch128")
    p.add_argument("--assets", type=int, default=128,
                   help="assets per GPU (the batch128 workload's sweep axis; default its largest point)")
    p.add_argument("--sweep", default="1,8,16,32,64",
                   help="smaller batch sizes timed on a prefix of the batch ('' to skip)")
    p.add_argument("--corr", default="sparse", choices=["sparse", "mask", "geometry", "table"])
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--no-raster", action="store_true", help="skip the position-map rasteriser measurement")
    p.add_argument("--no-workloads", action="store_true",
                   help="skip the other workloads' cached-step measurements (ring12_128, per-asset latency)")
    p.add_argument("--cpu-assets", type=int, default=32,
                   help="assets in the oracle's timed sample for cpu_baseline (one trajectory, ~10-30 s)")
    p.add_argument("--ref-assets", type=int, default=2,
                   help="assets per step of the reference arm (the oracle; one trajectory each, ~1 s)")
    return p.parse_args()


# ------------------------------------------------------------------ setup --
def reduce_max(x: float, world: int) -> float:
    """Maximum of a float over all ranks (gloo; no collective on the data path)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(pixels_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput: every rank processes its own assets (weak
    scaling), the job takes as long as the slowest rank."""
    return pixels_per_rank * world / seconds


def dist_env():
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local = int(os.environ.get("LOCAL_RANK", 0))
    return rank, world, local


def workload(args, rank=0):
    """This rank's shard of the job's assets: global assets rank*B .. rank*B + B - 1
    (B = --assets per GPU; weak scaling), each rendered from its own seed."""
    from paper_2608_13255_gb300 import synth
    return synth.make_workload(args.workload, B=args.assets, first_asset=rank * args.assets)


def describe(w):
    return ("%s: %d assets x %d views, %dx%dx%d %s latents + f32 x0 cache, %d rotating anchors, "
            "%d-step %s, schedule %s, K=%d" % (w.name, w.B, w.N, w.H, w.W, w.C, w.dtype, w.a, w.S,
                                              w.sampler.upper(), json.dumps(w.schedule), w.K))


def step_bytes(w, B=None):
    """Algorithmic HBM bytes of one cached transport step (latents only) of B
    assets (default: the workload's):
    non-anchor element: x0_prev 4 + x0 write 4 + x_t 2 + x_next 2 (bf16) = 12 B;
    anchor element: x0_new 4 + x0_prev 4 (for the increment) + cache write 4 + 4 (latents) = 16 B."""
    B = w.B if B is None else B
    lb = 2 if w.dtype == "bf16" else 4
    hw = w.H * w.W
    non = B * (w.N - w.a) * w.C * hw * (8 + 2 * lb)
    anc = B * w.a * w.C * hw * (12 + 2 * lb)
    return non + anc


def measure_stages(traj, reps=20):
    """Graph-replay time of the trajectory's other stages: the correspondence
    build (tau, keep masks and tile counts, offsets, records) and one full
    step (the sampler reconstruction of every view from the denoiser's x0:
    x_t and x0 read, x_{t-1} written, 4 + 2 * 2 bytes per bf16 element)."""
    import torch
    w = traj.w
    full_t = next(t for t in range(w.S) if t not in traj.anchor_x0)
    lb = 2 if w.dtype == "bf16" else 4
    out = {}
    for name, g, nbytes in (("build", traj.g_build, None),
                            ("full_step", traj.g_steps[full_t], w.B * w.N * w.C * w.H * w.W * (4 + 2 * lb))):
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            g.replay()
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1) * 1e3)
        us = statistics.median(ts)
        out[name] = {"us": us}
        if nbytes:
            out[name].update({"alg_bytes": nbytes, "GBs": nbytes / us / 1e3,
                              "frac_of_peak": nbytes / us / 1e3 / measured_peak()[0]})
    out["what"] = "median of %d graph replays, %d assets" % (reps, w.B)
    return out


def measure_ablations(traj, reps=24):
    """Cached-step time of the two ablation modes of Sec. 4.3 (value copy,
    shuffled correspondence) beside the delta transport, on the bench's
    workload and first cached anchor set: each graph runs `reps` steps
    ping-ponging the x0 cache (every step reads and writes more than the L2
    holds).  Sparse mode only."""
    import torch
    from paper_2608_13255_gb300 import synth
    gc, w = traj.gc, traj.w
    t0 = next(iter(traj.anchor_x0))
    anchors = sorted(gc.rotate_anchors(w.N, w.a, t0, w.S, traj.sched)[0])
    T = gc.tiles_per_view(w.H, w.W)
    tp = traj.corr._keep["tile_ptr"].cpu().numpy().astype(np.int64)
    perm = torch.from_numpy(synth.pair_permutation(tp[T::T] - tp[:-1:T], seed=1)).to(traj.dev)
    shuffled = gc.permute_records(traj.corr, perm)
    hw, lb = w.H * w.W, (2 if w.dtype == "bf16" else 4)
    variants = (("delta", traj.corr, "delta", step_bytes(w)),
                ("value_copy", traj.corr, "copy", step_bytes(w) - w.B * w.a * w.C * hw * 4),
                ("shuffled", shuffled, "delta", step_bytes(w)))
    out = {}
    for name, corr, update, nbytes in variants:
        def one(i):
            src, dst = traj.bufs[i % 2], traj.bufs[(i + 1) % 2]
            gc.transport_step(corr, anchors, w.C, traj.anchor_x0[t0], src, dst, traj.x, traj.x, traj.recon[t0],
                              workspace=traj.workspace, update=update)
        for i in range(2):
            one(i)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(reps):
                one(i)
        g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / reps
        out[name] = {"us_per_step": us, "alg_bytes": nbytes, "GBs": nbytes / us / 1e3,
                     "frac_of_peak": nbytes / us / 1e3 / measured_peak()[0]}
    gc.device_status()
    out["what"] = ("one cached step, %d assets, anchors %s, %d steps per graph; value_copy reads no anchor "
                   "x0(t-1); shuffled = records permuted within each (b, v, u) pair (seed 1)" % (w.B, anchors, reps))
    return out


def measure_sweep(traj, sizes, reps=24):
    """Cached-step time against the number of assets per launch (the
    workload's batch sweep): for each size the first B' assets of the bench's
    batch get their own correspondence build and one graph of `reps` delta
    steps ping-ponging the x0 cache (first cached anchor set).  Below about
    25 assets a step's bytes fit in the 129 MB L2, so the fraction of the HBM
    peak is not a DRAM figure there."""
    import torch
    gc, w = traj.gc, traj.w
    t0 = next(iter(traj.anchor_x0))
    anchors = sorted(gc.rotate_anchors(w.N, w.a, t0, w.S, traj.sched)[0])
    peak = measured_peak()[0]
    out = {}
    for bs in sorted(set(sizes) | {w.B}):
        if bs < 1 or bs > w.B:
            continue
        if bs == w.B:
            corr, wsp = traj.corr, traj.workspace
        else:
            corr = gc.build_sparse_corr(traj.pos[:bs], traj.valid[:bs], traj.cams[:bs], K=w.K, tol_frac=w.tol_frac)
            wsp = torch.empty(max(corr.workspace_floats(w.C), 4), dtype=torch.float32, device=traj.dev)
        new, x, bufs = traj.anchor_x0[t0][:bs], traj.x[:bs], [b[:bs] for b in traj.bufs]

        def one(i):
            gc.transport_step(corr, anchors, w.C, new, bufs[i % 2], bufs[(i + 1) % 2], x, x, traj.recon[t0],
                              workspace=wsp)
        for i in range(2):
            one(i)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(reps):
                one(i)
        g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / reps
        nbytes = step_bytes(w, bs)
        out[str(bs)] = {"us_per_step": us, "alg_bytes": nbytes, "frac_of_peak": nbytes / us / 1e3 / peak,
                        "target_pixels_per_s": bs * (w.N - w.a) * w.H * w.W / us * 1e6}
        del g, corr
    gc.device_status()
    out["what"] = ("one cached delta step on the first B' assets, %d steps per graph, anchors %s; keys are B'"
                   % (reps, anchors))
    return out


def time_cached_steps(w, B, dev, reps=24, seed=3, cold=False):
    """One graph of `reps` cached transport steps of workload w replicated to
    B assets (its own correspondence build, sparse mode), the anchor set
    rotating as the workload's schedule rotates it over its cached steps and
    the x0 cache ping-ponging between two buffers; latents in place.
    Returns (us per step, algorithmic bytes per step, target view-pixels per
    step, anchor sets, cold us per step or None).  cold: also time single
    steps (one graph each) with the L2 flushed before each, outside the timed
    region (a 256 MB buffer written), as a step meets it after a denoiser
    forward."""
    import torch
    from paper_2608_13255_gb300 import geocache as gc
    from paper_2608_13255_gb300 import synth
    wb = synth.replicate_assets(w, B)
    pos, valid, cams = (torch.from_numpy(a).to(dev) for a in (wb.pos, wb.valid, wb.cams))
    corr = gc.build_sparse_corr(pos, valid, cams, K=wb.K, tol_frac=wb.tol_frac)
    wsp = torch.empty(max(corr.workspace_floats(wb.C), 4), dtype=torch.float32, device=dev)
    cached = [t for t in range(wb.S) if not gc.rotate_anchors(wb.N, wb.a, t, wb.S, wb.schedule)[1]]
    sets = []
    for t in cached:
        a = tuple(gc.rotate_anchors(wb.N, wb.a, t, wb.S, wb.schedule)[0])
        if a not in sets:
            sets.append(a)
    g0 = torch.Generator(device=dev).manual_seed(seed)
    shp = (B, wb.N, wb.C, wb.H, wb.W)
    bufs = [torch.randn(shp, device=dev, generator=g0) for _ in range(2)]
    lat = torch.bfloat16 if wb.dtype == "bf16" else torch.float32
    x = torch.randn(shp, device=dev, generator=g0).to(lat)
    new = {a: torch.randn((B, wb.a, wb.C, wb.H, wb.W), device=dev, generator=g0) for a in sets}
    p = synth.recon_params(wb, cached[0])
    r = gc.make_recon(p["sampler"], a_t=p.get("a_t", 0), a_prev=p.get("a_prev", 0), sigma=p.get("sigma", 0),
                      sigma_next=p.get("sigma_next", 0))

    def one(i):
        a = sets[i % len(sets)]
        gc.transport_step(corr, list(a), wb.C, new[a], bufs[i % 2], bufs[(i + 1) % 2], x, x, r, workspace=wsp)
    for i in range(2):
        one(i)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for i in range(reps):
            one(i)
    g.replay()
    ts = []
    for _ in range(3):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1) * 1e3 / reps)
    gc.device_status()
    us = statistics.median(ts)
    us_cold = None
    if cold:
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        singles = []
        for i in range(2):
            gs = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gs):
                one(i)
            singles.append(gs)
        tc = []
        for k in range(20):
            flush.fill_(k & 0xff)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            singles[k % 2].replay()
            e1.record()
            torch.cuda.synchronize()
            tc.append(e0.elapsed_time(e1) * 1e3)
        gc.device_status()
        us_cold = statistics.median(tc)
        del flush
    return us, step_bytes(wb), B * (wb.N - wb.a) * wb.H * wb.W, sets, us_cold


def measure_workloads(dev, reps=24):
    """Cached-step times of the other workloads (sparse mode, 24-step graphs,
    anchors rotating as each workload's schedule rotates them):
    * ring12_128 (12 views, 128 x 128 x 16 bf16, 4 anchors, FM-Euler)
      replicated to 8 assets (335 MB per step, more than the L2): a DRAM
      figure against the measured copy peak;
    * the paper's per-asset regime, one asset per step (hunyuan64,
      solids96, ring12_128) and batch128 at its base batch of 8 assets:
      these steps fit in the 129 MB L2, so they are reported as latency."""
    from paper_2608_13255_gb300 import synth
    peak = measured_peak()[0]
    out = {}
    r12 = synth.make_workload("ring12_128")
    for name, w, B in (("ring12_128_x8", r12, 8), ("ring12_128_x1", r12, 1),
                       ("hunyuan64_x1", synth.make_workload("hunyuan64"), 1),
                       ("solids96_x1", synth.make_workload("solids96"), 1),
                       ("batch128_x8", synth.make_workload("batch128", B=8), 8)):
        small = step_bytes(synth.replicate_assets(w, B)) <= L2_BYTES
        us, nbytes, pix, sets, us_cold = time_cached_steps(w, B, dev, reps, cold=small)
        d = {"us_per_step": us, "alg_bytes": nbytes, "target_pixels_per_s": pix / us * 1e6,
             "anchor_sets": [list(a) for a in sets]}
        if nbytes > L2_BYTES:
            d["frac_of_peak"] = nbytes / us / 1e3 / peak
        else:
            d["fits_in_l2"] = True
            d["us_per_step_cold"] = us_cold
        out[name] = d
    out["what"] = ("one cached step (sparse mode) per graph node, %d steps per graph, median of 3 replays; "
                   "frac_of_peak only where a step moves more than the L2 holds; for steps that fit in the "
                   "L2, us_per_step_cold: one step per graph replay with the L2 flushed before it (a 256 MB "
                   "buffer written outside the timed region), median of 20" % reps)
    return out


def measure_raster(dev, B, N_layout, H, W, reps=10, cpu_assets=2):
    """Position maps of B meshes (icosphere subdivision 6 with smooth radial
    noise: 40962 vertices, 81920 faces; four distinct meshes tiled over the
    batch) seen by the workload's N cameras (azimuths offset per asset), at
    H x W: GPU time of one geocache_raster_posmaps call (z-buffer clear,
    face kernel, resolve kernel) and the oracle's single-threaded time on
    `cpu_assets` of the assets."""
    import torch
    import oracle
    from paper_2608_13255_gb300 import geocache as gc
    from paper_2608_13255_gb300 import synth
    base = [synth.blob_mesh(6, 0.15, np.random.default_rng(100 + k)) for k in range(4)]
    meshes = [(base[b % 4][0].astype(np.float32), base[b % 4][1].astype(np.int32)) for b in range(B)]
    cams = np.stack([np.stack([synth.look_at_camera(az + 7.0 * b, el, H, W) for az, el in N_layout])
                     for b in range(B)])
    v_off = np.cumsum([0] + [len(V) for V, _ in meshes])
    f_off = torch.from_numpy(np.cumsum([0] + [len(F) for _, F in meshes]).astype(np.int64)).to(dev)
    verts = torch.from_numpy(np.concatenate([V for V, _ in meshes])).to(dev)
    faces = torch.from_numpy(np.concatenate([F + v_off[b] for b, (_, F) in enumerate(meshes)]).astype(np.int32)).to(dev)
    d_cams = torch.from_numpy(cams).to(dev)
    N = len(N_layout)
    zbuf = torch.empty((B, N, H, W), dtype=torch.int64, device=dev)
    pos = torch.empty((B, N, H, W, 3), dtype=torch.float32, device=dev)
    valid = torch.empty((B, N, H, W), dtype=torch.uint8, device=dev)
    for _ in range(2):
        gc.raster_posmaps(verts, faces, f_off, d_cams, H, W, zbuf, pos, valid)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        gc.raster_posmaps(verts, faces, f_off, d_cams, H, W, zbuf, pos, valid)
    e1.record()
    torch.cuda.synchronize()
    gc.device_status()
    us = e0.elapsed_time(e1) * 1e3 / reps
    pixels, face_views = B * N * H * W, N * int(faces.shape[0])
    t0 = time.perf_counter()
    for b in range(cpu_assets):
        oracle.raster_views(meshes[b][0], meshes[b][1], cams[b], H, W)
    cpu_s = time.perf_counter() - t0
    return {"what": "%d meshes x %d views at %dx%d, 81920 faces each" % (B, N, H, W),
            "us_per_batch": us, "pixels_per_s": pixels / us * 1e6, "face_views_per_s": face_views / us * 1e6,
            "covered_frac": float(valid.float().mean()), "launches_per_call": 2,
            "cpu_oracle": {"pixels_per_s": cpu_assets * N * H * W / cpu_s, "cores": 1,
                           "sample": "%d of the meshes, all views" % cpu_assets}}


def measure_supersampled(dev, B=16, H=128, W=128, s=4, reps=5):
    """Position maps rendered at s times the token grid and pooled to it
    (geocache_raster_posmaps_supersampled: the image-resolution render of a
    pipeline, 512 x 512 for 128 x 128 tokens at s = 4), and the pooling alone
    of caller-rendered fine maps (geocache_pool_posmaps, HBM-bound: 13 B read
    per fine pixel, 13 B written per token).  B meshes of the rasteriser
    measurement, the workload's 6 cameras."""
    import torch
    from paper_2608_13255_gb300 import geocache as gc
    from paper_2608_13255_gb300 import synth
    base = [synth.blob_mesh(6, 0.15, np.random.default_rng(100 + k)) for k in range(4)]
    meshes = [(base[b % 4][0].astype(np.float32), base[b % 4][1].astype(np.int32)) for b in range(B)]
    layout = synth.hunyuan_layout()
    cams = np.stack([np.stack([synth.look_at_camera(az + 7.0 * b, el, H, W) for az, el in layout]) for b in range(B)])
    v_off = np.cumsum([0] + [len(V) for V, _ in meshes])
    f_off = torch.from_numpy(np.cumsum([0] + [len(F) for _, F in meshes]).astype(np.int64)).to(dev)
    verts = torch.from_numpy(np.concatenate([V for V, _ in meshes])).to(dev)
    faces = torch.from_numpy(np.concatenate([F + v_off[b] for b, (_, F) in enumerate(meshes)]).astype(np.int32)).to(dev)
    d_cams = torch.from_numpy(cams).to(dev)
    N = len(layout)
    zbuf = torch.empty((B, N, s * H, s * W), dtype=torch.int64, device=dev)
    pos = torch.empty((B, N, H, W, 3), dtype=torch.float32, device=dev)
    valid = torch.empty((B, N, H, W), dtype=torch.uint8, device=dev)

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / reps
    us_ss = timed(lambda: gc.raster_posmaps(verts, faces, f_off, d_cams, H, W, zbuf, pos, valid, s=s))
    # fine maps rendered directly at s x (cameras scaled), then pooled
    cams_hi = d_cams.clone()
    cams_hi[..., 12:16] *= s
    fine_p = torch.empty((B, N, s * H, s * W, 3), dtype=torch.float32, device=dev)
    fine_v = torch.empty((B, N, s * H, s * W), dtype=torch.uint8, device=dev)
    gc.raster_posmaps(verts, faces, f_off, cams_hi, s * H, s * W, zbuf, fine_p, fine_v)
    pos2, valid2 = torch.empty_like(pos), torch.empty_like(valid)
    us_pool = timed(lambda: gc.pool_posmaps(fine_p, fine_v, s, pos2, valid2))
    torch.cuda.synchronize()
    gc.device_status()
    same = bool(torch.equal(valid, valid2) and torch.equal(pos.view(torch.int32), pos2.view(torch.int32)))
    fine_px = B * N * s * s * H * W
    pool_bytes = fine_px * 13 + B * N * H * W * 13
    return {"what": "%d meshes x %d views, %dx%d tokens rendered at %dx%d (s = %d), 81920 faces each"
                    % (B, N, H, W, s * H, s * W, s),
            "raster_supersampled_us": us_ss, "fine_pixels_per_s": fine_px / us_ss * 1e6,
            "pool_us": us_pool, "pool_alg_bytes": pool_bytes, "pool_GBs": pool_bytes / us_pool / 1e3,
            "pool_frac_of_peak": pool_bytes / us_pool / 1e3 / measured_peak()[0],
            "pooled_equals_fused": same}


def step_runs(S, cached_steps):
    """The graphs of one trajectory: (first step, end step, cached, head) per
    run of consecutive sampler steps of one kind, in order.  head marks a run
    of full steps that opens the trajectory: full steps read no
    correspondence, so the build runs beside them on a side stream of the same
    graph, joined before the first cached step."""
    runs, t = [], 0
    while t < S:
        cached = t in cached_steps
        u = t
        while u < S and (u in cached_steps) == cached:
            u += 1
        runs.append((t, u, cached, t == 0 and not cached))
        t = u
    return runs


class Trajectory:
    """Device state of one batch's trajectory and the loop over its steps."""

    def __init__(self, w, dev, corr_mode="sparse"):
        import torch
        from paper_2608_13255_gb300 import geocache as gc
        from paper_2608_13255_gb300 import synth
        self.gc, self.w, self.dev = gc, w, dev
        self.sched = w.schedule
        self.pos = torch.from_numpy(w.pos).to(dev)
        self.valid = torch.from_numpy(w.valid).to(dev)
        self.cams = torch.from_numpy(w.cams).to(dev)
        self.tau = torch.zeros(w.B, dtype=torch.float32, device=dev)
        idx = wt = keep = tile_ptr = records = None
        if corr_mode == "table":
            shp = (w.B, w.N, w.N, w.H, w.W, w.K)
            idx = torch.empty(shp, dtype=torch.int32, device=dev)
            wt = torch.empty(shp, dtype=torch.float32, device=dev)
        if corr_mode in ("mask", "sparse"):
            keep = torch.empty((w.B, w.N, w.N, w.H, w.W), dtype=torch.uint8, device=dev)
        src_ptr = src_rec = None
        if corr_mode == "sparse":
            tile_ptr = torch.empty(w.B * w.N * w.N * gc.tiles_per_view(w.H, w.W) + 1, dtype=torch.int32, device=dev)
            c0 = gc.make_corr(self.pos, self.valid, self.cams, self.tau, K=w.K, tol_frac=w.tol_frac, keep=keep,
                              tile_ptr=tile_ptr, mode=gc.CORR_MASK)
            records = torch.empty((max(gc.record_count(c0), 1), 4), dtype=torch.int32, device=dev)
        mode = {"mask": gc.CORR_MASK, "table": gc.CORR_TABLE, "geometry": gc.CORR_GEOMETRY,
                "sparse": gc.CORR_SPARSE}[corr_mode]
        self.corr = gc.make_corr(self.pos, self.valid, self.cams, self.tau, idx, wt, K=w.K, tol_frac=w.tol_frac,
                                 mode=mode, keep=keep, tile_ptr=tile_ptr, records=records, src_ptr=src_ptr,
                                 src_rec=src_rec)
        nws = self.corr.workspace_floats(w.C)
        self.workspace = torch.empty(max(nws, 4), dtype=torch.float32, device=dev) if nws else None
        xT, x0 = synth.initial_latents(w)
        lat = torch.bfloat16 if w.dtype == "bf16" else torch.float32
        self.x = torch.from_numpy(xT).to(dev).to(lat)
        x0_d = torch.from_numpy(x0).to(dev)
        self.full_x0, self.anchor_x0, self.recon = {}, {}, {}
        for t in range(w.S):
            p = synth.recon_params(w, t)
            self.recon[t] = gc.make_recon(p["sampler"], a_t=p.get("a_t", 0), a_prev=p.get("a_prev", 0),
                                          sigma=p.get("sigma", 0), sigma_next=p.get("sigma_next", 0))
            anchors, full = gc.rotate_anchors(w.N, w.a, t, w.S, self.sched)
            if full:
                d = torch.from_numpy(synth.delta(w, t, list(range(w.N)))).to(dev)
                self.full_x0[t] = (x0_d + d).contiguous()
            else:
                d = torch.from_numpy(synth.delta(w, t, anchors)).to(dev)
                self.anchor_x0[t] = (x0_d[:, anchors] + d).contiguous()
        self.bufs = [torch.empty_like(x0_d), torch.empty_like(x0_d)]
        self.n_cached = len(self.anchor_x0)
        self.anchor_sets = {tuple(gc.rotate_anchors(w.N, w.a, t, w.S, self.sched)[0]) for t in self.anchor_x0}
        self.pixels = self.n_cached * w.B * (w.N - w.a) * w.H * w.W

    def host_inputs(self):
        """Pinned host copies of every input of one trajectory (for e2e)."""
        import torch
        pin = lambda t: t.cpu().pin_memory()
        return {"pos": pin(self.pos), "valid": pin(self.valid), "cams": pin(self.cams), "x": pin(self.x),
                "full": {t: pin(v) for t, v in self.full_x0.items()},
                "anchor": {t: pin(v) for t, v in self.anchor_x0.items()}}

    def run(self, events=None):
        """Enqueue one trajectory eagerly; returns the number of kernels launched.
        events: list receiving (start, end, 1) CUDA events around each cached step."""
        import torch
        gc, w = self.gc, self.w
        launches = 0
        gc.build_corr(self.corr)
        launches += 1 + (1 if (self.corr.idx is not None or self.corr.keep is not None) else 0)
        if self.corr.c.mode == gc.CORR_SPARSE:
            launches += 2  # the tile offsets' scan, the records
            if self.corr.c.src_ptr:
                launches += 3  # the source index: counts, their scan, the scatter
        cache = None
        for t in range(w.S):
            timed = events is not None and t in self.anchor_x0
            if timed:
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
            cache, n = self._step(t, cache)
            launches += n
            if timed:
                e1.record()
                events.append((e0, e1, 1))
        self.launches = launches
        return launches

    def _step(self, t, cache):
        """Enqueue sampler step t; returns (new cache, kernels launched)."""
        gc, w = self.gc, self.w
        anchors, full = gc.rotate_anchors(w.N, w.a, t, w.S, self.sched)
        if full:
            gc.reconstruct(self.x, self.full_x0[t], self.x, self.recon[t])
            return self.full_x0[t], 1
        out = self.bufs[0] if cache is not self.bufs[0] else self.bufs[1]
        gc.transport_step(self.corr, anchors, w.C, self.anchor_x0[t], cache, out, self.x, self.x, self.recon[t],
                          workspace=self.workspace)
        return out, gc.transport_launches(w.a, w.N, self.corr.c.mode, in_place=False)

    def capture(self):
        """Capture the correspondence build and every sampler step in CUDA
        graphs; False (and eager launches) if capture is unavailable."""
        import torch
        self.run()  # lazy initialisation outside capture
        torch.cuda.synchronize()
        try:
            self.g_build = torch.cuda.CUDAGraph()
            with torch.cuda.graph(self.g_build):
                self.gc.build_corr(self.corr)
            # one graph per sampler step (the e2e path waits for each step's
            # uploads), and one per run of consecutive steps of one kind (full
            # or cached: the timed trajectories)
            self.g_steps = []
            cache = None
            for t in range(self.w.S):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    cache, _ = self._step(t, cache)
                self.g_steps.append(g)
            self.g_runs = []
            self.build_in_head = False
            side = torch.cuda.Stream()
            cache = None
            for t, u, cached, head in step_runs(self.w.S, set(self.anchor_x0)):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    if head:
                        cur = torch.cuda.current_stream()
                        side.wait_stream(cur)
                        with torch.cuda.stream(side):
                            self.gc.build_corr(self.corr)
                    for k in range(t, u):
                        cache, _ = self._step(k, cache)
                    if head:
                        cur.wait_stream(side)
                self.build_in_head = self.build_in_head or head
                self.g_runs.append((g, cached, u - t))
            self.replay(None)
            torch.cuda.synchronize()
        except RuntimeError as exc:
            print("bench: CUDA graph capture failed (%s); timing eager launches" % exc, file=sys.stderr)
            self.g_build = self.g_steps = self.g_runs = None
            return False
        return True

    def replay(self, events=None):
        """Replay one trajectory: the build (inside the first run's graph when
        the trajectory opens with full steps), then each run of full or cached
        steps.  events: list receiving (start, end, steps) CUDA events around
        each run of cached steps."""
        import torch
        if not self.build_in_head:
            self.g_build.replay()
        for g, cached, n in self.g_runs:
            timed = events is not None and cached
            if timed:
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
            g.replay()
            if timed:
                e1.record()
                events.append((e0, e1, n))

    def run_e2e(self, host, graph=None):
        """One trajectory from pinned host inputs to a host copy of the final
        latents (the trajectory itself replayed from `graph` when given).
        With graphs the uploads run on a copy stream in the order the steps
        need them and each step waits only for its own inputs, so compute
        overlaps the remaining uploads."""
        import torch
        if graph:
            return self._run_e2e_overlapped(host)
        self.pos.copy_(host["pos"], non_blocking=True)
        self.valid.copy_(host["valid"], non_blocking=True)
        self.cams.copy_(host["cams"], non_blocking=True)
        self.x.copy_(host["x"], non_blocking=True)
        for t, v in host["full"].items():
            self.full_x0[t].copy_(v, non_blocking=True)
        for t, v in host["anchor"].items():
            self.anchor_x0[t].copy_(v, non_blocking=True)
        if graph:
            self.replay()
        else:
            self.run()
        out = self._host_out()
        out.copy_(self.x, non_blocking=True)
        torch.cuda.current_stream().synchronize()
        return out

    def _host_out(self):
        """Pinned host buffer of the final latents, allocated once."""
        import torch
        if getattr(self, "host_out", None) is None:
            self.host_out = torch.empty(self.x.shape, dtype=self.x.dtype, pin_memory=True)
        return self.host_out

    def _run_e2e_overlapped(self, host):
        import torch
        cur = torch.cuda.current_stream()
        if getattr(self, "copy_stream", None) is None:
            self.copy_stream = torch.cuda.Stream()
        cs = self.copy_stream
        cs.wait_stream(cur)  # the previous trajectory is done with these buffers
        ready = []
        with torch.cuda.stream(cs):
            for name in ("pos", "valid", "cams", "x"):
                getattr(self, name).copy_(host[name], non_blocking=True)
            ready.append(torch.cuda.Event())
            ready[-1].record(cs)
            for t in range(self.w.S):
                if t in host["full"]:
                    self.full_x0[t].copy_(host["full"][t], non_blocking=True)
                if t in host["anchor"]:
                    self.anchor_x0[t].copy_(host["anchor"][t], non_blocking=True)
                ready.append(torch.cuda.Event())
                ready[-1].record(cs)
        cur.wait_event(ready[0])
        self.g_build.replay()
        for t, g in enumerate(self.g_steps):
            cur.wait_event(ready[t + 1])
            g.replay()
        out = self._host_out()
        out.copy_(self.x, non_blocking=True)
        cur.synchronize()
        return out

    def h2d_bytes(self):
        n = lambda t: t.numel() * t.element_size()
        return (n(self.pos) + n(self.valid) + n(self.cams) + n(self.x) + sum(n(v) for v in self.full_x0.values())
                + sum(n(v) for v in self.anchor_x0.values()))

    def working_set(self):
        n = lambda t: t.numel() * t.element_size()
        return 2 * n(self.x) + 2 * n(self.bufs[0]) + n(next(iter(self.anchor_x0.values())))


# ----------------------------------------------------------------- clocks --
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        # raw samples (nvidia-smi CSV) beside the run's other scratch output
        self.path = os.path.join(os.environ.get("BENCH_CLOCKS_DIR", tempfile.gettempdir()),
                                 "geocache_clocks_rank%d.csv" % gpu_index)

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def measured_traffic(kernel_hash, assets, workload):
    """DRAM bytes of one transport step from the committed ncu summary of
    `workload`, scaled to `assets`; None when the kernels changed since the
    capture or no summary covers the workload."""
    path = os.path.join(ROOT, "profiles", "transport_traffic.txt")
    try:
        kv = dict(line.split() for line in open(path) if line.strip() and not line.startswith("#"))
        if kv.get("kernel_hash") != kernel_hash or kv.get("workload") != workload:
            return None
        return float(kv["bytes_per_step"]) * assets / float(kv["assets"])
    except (OSError, ValueError, KeyError):
        return None


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


# ------------------------------------------------------------ CPU oracle --
def oracle_trajectory(w, steps=None, state=False):
    """The CPU oracle, as it stands, over one trajectory of workload w.
    Returns (cached target view-pixels processed, seconds), plus the final
    latents and x0 cache when state is true."""
    import oracle
    from paper_2608_13255_gb300 import synth
    t0 = time.perf_counter()
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    geom = (w.pos, w.valid, w.cams, tau)
    xT, x0 = synth.initial_latents(w)
    x = xT.astype(np.float64)
    cache = x0.astype(np.float64)
    pixels = 0
    S = w.S if steps is None else steps
    for t in range(S):
        p = synth.recon_params(w, t)
        rk = dict(sampler=oracle.DDIM if p["sampler"] == "ddim" else oracle.FM_EULER, a_t=p.get("a_t", 0.0),
                  a_prev=p.get("a_prev", 0.0), sigma=p.get("sigma", 0.0), sigma_next=p.get("sigma_next", 0.0))
        if oracle.is_full_step(t, w.S, w.schedule):
            cache = cache + synth.delta(w, t, list(range(w.N)))
            x, _ = oracle.reconstruct(x, cache, **rk)
        else:
            anchors = oracle.rotate_anchors(w.N, w.a, oracle.cached_ordinal(t, w.S, w.schedule))
            new = cache[:, anchors] + synth.delta(w, t, anchors)
            cache, x, _ = oracle.transport_step(anchors, new, cache, geom=geom, x_t=x, recon=rk)
            pixels += w.B * (w.N - w.a) * w.H * w.W
        if w.dtype == "bf16":
            x = (oracle.round_bf16(x).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    if state:
        return pixels, time.perf_counter() - t0, x, cache
    return pixels, time.perf_counter() - t0


def cpu_baseline(args, w_full):
    from paper_2608_13255_gb300 import synth
    ws = synth.replicate_assets(w_full, args.cpu_assets)
    pixels, secs = oracle_trajectory(ws)
    return {"value": pixels / secs, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": "%d of the %d assets, one whole %d-step trajectory (%.1f s, single-threaded C oracle)" % (
                args.cpu_assets, w_full.B, w_full.S, secs)}


def _asset_subset(w, idx):
    """Workload w restricted to the contiguous assets idx (same recipe, fewer assets)."""
    idx = np.asarray(idx)
    assert len(idx) and (np.diff(idx) == 1).all(), "asset subsets are contiguous ranges"
    out = type(w)(**{**w.__dict__})
    out.B = len(idx)
    out.first_asset = w.first_asset + int(idx[0])
    out.cams = np.ascontiguousarray(w.cams[idx])
    out.pos = np.ascontiguousarray(w.pos[idx])
    out.valid = np.ascontiguousarray(w.valid[idx])
    return out


def _oracle_worker(w, barrier, queue):
    """One process of the all-cores CPU baseline: the unchanged oracle over
    its share of the assets, timed from a barrier shared by all workers."""
    try:
        import oracle  # noqa: F401  (loads the C core before the clock starts)
        barrier.wait(timeout=300)
        t0 = time.time()
        pixels, _ = oracle_trajectory(w)
        queue.put((pixels, t0, time.time()))
    except Exception as exc:  # reported by the parent
        queue.put(("error", repr(exc), 0.0))


def cpu_baseline_all_cores(w_full, cores=None):
    """The oracle, as it stands, on every asset of the workload with one
    process per host core (assets are independent, so they split with no
    communication); value = all cached target view-pixels / wall time from
    the common start to the last worker's end.  Processes are spawned (CUDA
    is already initialised in this one)."""
    import multiprocessing as mp
    cores = max(1, min(cores or os.cpu_count() or 1, w_full.B))
    ctx = mp.get_context("spawn")
    barrier, queue = ctx.Barrier(cores), ctx.Queue()
    parts = np.array_split(np.arange(w_full.B), cores)
    procs = [ctx.Process(target=_oracle_worker, args=(_asset_subset(w_full, idx), barrier, queue)) for idx in parts]
    for p in procs:
        p.start()
    import queue as queue_mod
    res, t_end = [], time.time() + 900
    while len(res) < len(procs):
        try:
            res.append(queue.get(timeout=5))
        except queue_mod.Empty:
            if time.time() > t_end or not any(p.is_alive() for p in procs):
                for p in procs:
                    if p.is_alive():
                        p.terminate()
                raise RuntimeError("oracle workers ended with %d of %d results" % (len(res), len(procs)))
    for p in procs:
        p.join(timeout=60)
    bad = [r for r in res if r[0] == "error"]
    if bad:
        raise RuntimeError("oracle worker failed: %s" % bad[0][1])
    pixels = sum(r[0] for r in res)
    wall = max(r[2] for r in res) - min(r[1] for r in res)
    return {"value": pixels / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "all %d assets, one whole %d-step trajectory, %d processes of the single-threaded C oracle "
                      "(%.1f s wall)" % (w_full.B, w_full.S, cores, wall)}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2608_13255_gb300 import synth
    w = workload(args)
    ws = synth.replicate_assets(w, args.ref_assets)
    for _ in range(args.warmup):
        oracle_trajectory(ws, steps=6)
    tot_pix, tot_s = 0, 0.0
    for _ in range(args.steps):
        pix, s = oracle_trajectory(ws)
        tot_pix += pix
        tot_s += s
    value = tot_pix / tot_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": describe(w), "sampled_assets": args.ref_assets},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": "%d of %d assets per step, whole trajectories" % (args.ref_assets, w.B)},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------------- main --
def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    import torch
    import torch.distributed as dist
    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("gloo")
    torch.cuda.set_device(local)
    dev = "cuda:%d" % local
    from paper_2608_13255_gb300 import build as gbuild
    gbuild.build()
    w = workload(args, rank)
    traj = Trajectory(w, dev, args.corr)
    ws_bytes = traj.working_set()

    def barrier():
        if world > 1:
            dist.barrier()

    # every kernel launch of a trajectory is captured once in CUDA graphs (one
    # for the correspondence build, one per run of consecutive full or cached
    # sampler steps) and replayed, so launches cost no host time; events
    # between the replays time each run of cached steps' transport kernels
    events = []
    use_graphs = traj.capture()
    launches_per_traj = traj.launches

    def one_step(ev=None):
        if use_graphs:
            traj.replay(ev)
        else:
            traj.run(ev)
        return launches_per_traj

    args.warmup = max(3, args.warmup)  # at least three untimed warm-up steps
    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize()

    launches = 0
    with ClockSampler(local) as clocks:
        barrier()
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        # an NVTX range around the timed trajectories lets a profiler list
        # exactly their launches (ncu --nvtx --nvtx-include "timed_trajectories/")
        torch.cuda.nvtx.range_push("timed_trajectories")
        for _ in range(args.steps):
            launches += one_step(events)
        torch.cuda.nvtx.range_pop()
        t1.record()
        torch.cuda.synchronize()
        barrier()
    ms = reduce_max(t0.elapsed_time(t1), world)
    kernel_ms = [(a.elapsed_time(b), n) for a, b, n in events]
    ms_per_step = ms / args.steps
    total_pixels = traj.pixels * world
    value = job_value(traj.pixels, world, ms_per_step / 1e3)

    k_launches = sum(n for _, n in kernel_ms)
    k_avg_ms = sum(ms for ms, _ in kernel_ms) / k_launches
    alg = step_bytes(w)
    achieved = alg / (k_avg_ms / 1e3) / 1e9
    peak, peak_src = measured_peak()
    traffic = measured_traffic(gbuild.source_hash(), w.B, w.name)

    # secondary: anchor-row pack of the latents and scatter back (the batch
    # slicing around the denoiser's anchor-only forward); four source / slice
    # pairs in rotation (267 MB per cycle, larger than L2) so that each call
    # reads from HBM; bytes = rows read + rows written
    pack = None
    if rank == 0:
        anchors0 = sorted(next(iter(traj.anchor_sets)))
        srcs = [traj.x.clone() for _ in range(4)]
        sls = [torch.empty((w.B, len(anchors0)) + tuple(traj.x.shape[2:]), dtype=traj.x.dtype, device=dev)
               for _ in range(4)]
        reps = 48
        for i in range(4):
            traj.gc.pack_anchors(srcs[i], sls[i], anchors0)
        torch.cuda.synchronize()
        res = {}
        for name, fn in (("pack", lambda i: traj.gc.pack_anchors(srcs[i % 4], sls[i % 4], anchors0)),
                         ("unpack", lambda i: traj.gc.unpack_anchors(sls[i % 4], srcs[i % 4], anchors0))):
            gpk = torch.cuda.CUDAGraph()  # launched from a graph: the copies, not the host, are timed
            with torch.cuda.graph(gpk):
                for i in range(reps):
                    fn(i)
            gpk.replay()
            p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            p0.record()
            gpk.replay()
            p1.record()
            torch.cuda.synchronize()
            us = p0.elapsed_time(p1) * 1e3 / reps
            nbytes = 2 * sls[0].numel() * sls[0].element_size()
            res[name] = {"us_per_call": us, "GBs": nbytes / us / 1e3,
                         "frac_of_peak": nbytes / us / 1e3 / measured_peak()[0]}
        pack = {"what": "anchor rows (%d of %d views) of the bf16 latents, %d assets" % (len(anchors0), w.N, w.B),
                **res}
        del srcs, sls

    ablations = measure_ablations(traj) if rank == 0 and args.corr == "sparse" else None
    sweep = None
    if rank == 0 and args.corr == "sparse" and use_graphs and args.sweep:
        sweep = measure_sweep(traj, [int(x) for x in args.sweep.split(",")])
    stages = measure_stages(traj) if rank == 0 and use_graphs else None
    workloads = measure_workloads(dev) if rank == 0 and use_graphs and not args.no_workloads else None
    raster = None
    if rank == 0 and not args.no_raster:
        from paper_2608_13255_gb300 import synth
        layout = synth.hunyuan_layout() if w.N == 6 else synth.ring8_polar4_layout()[:w.N]
        raster = measure_raster(dev, w.B, layout, w.H, w.W)
        raster["supersampled"] = measure_supersampled(dev)

    e2e = None
    if not args.no_e2e:
        host = traj.host_inputs()
        traj.run_e2e(host, use_graphs)
        barrier()
        t_s = time.perf_counter()
        for _ in range(args.steps):
            out = traj.run_e2e(host, use_graphs)
        e2e_s = reduce_max((time.perf_counter() - t_s) / args.steps, world)
        e2e = {"value": job_value(traj.pixels, world, e2e_s), "unit": UNIT, "h2d_bytes_per_step": traj.h2d_bytes(),
               "d2h_bytes_per_step": out.numel() * out.element_size(), "ms_per_step": 1e3 * e2e_s}

    if rank != 0:
        return 0
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": describe(w), "assets_per_gpu": w.B, "corr": args.corr,
                   "storage": "bf16 latents, f32 x0 cache" if w.dtype == "bf16" else "f32",
                   "l2": "inputs larger than L2: %.0f MB touched per cached step vs %d MB L2" % (
                       ws_bytes / 1e6, L2_BYTES // 2 ** 20),
                   "step": "tau + correspondence build + %d-step trajectory (%d cached transport steps, %d full "
                           "steps)" % (w.S, traj.n_cached, w.S - traj.n_cached),
                   "launch": ("CUDA graphs (each run of consecutive full or cached sampler steps; the build "
                              "beside the opening full steps on a side stream, else its own graph) replayed"
                              if use_graphs else "eager")},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_source": peak_src,
                     "kernel": "sparse_phase_a_kernel + sparse_phase_b_kernel (one cached step)",
                     "alg_bytes_per_launch": alg,
                     "avg_launch_us": 1e3 * k_avg_ms, "launches": k_launches,
                     "timed_by": ("events around each graph replay of a run of consecutive cached steps "
                                  "(graph launch included), divided by its steps"),
                     "frac_of_8TBs": achieved / 8000.0},
        "gpu_launches": launches,
        "pack_anchors": pack,
        "stages": stages,
        "ablations": ablations,
        "batch_sweep": sweep,
        "workloads": workloads,
        "raster_posmaps": raster,
        "clocks": clocks.summary(),
        "e2e": e2e,
    }
    if not args.no_cpu and world == 1:
        line["cpu_baseline"] = cpu_baseline(args, w)
        line["cpu_baseline_all_cores"] = cpu_baseline_all_cores(w)
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
