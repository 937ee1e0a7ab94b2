"""GPU parity of the two ablation modes of Sec. 4.3 (Table 3) against the CPU
oracle, through the C ABI: the value copy (geocache_transport_step_update
with GEOCACHE_UPDATE_COPY, every correspondence mode) and the shuffled
correspondence (geocache_permute_records, then a sparse-mode step).  Same
tolerances as the transport parity tests (gpu_helpers)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_13255_gb300 import synth

from gpu_helpers import (DeviceGeometry, assert_bf16_close, assert_f32_close, latent_values, recon_kw,
                         step_inputs)

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


def _gpu_step(gc, w, g, corr, anchors, params, update="delta", step=3):
    x0_prev, x0_new, xt32 = step_inputs(w, step, anchors)
    xt64, xt_t = latent_values(xt32, w)
    d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
    d_out = torch.empty_like(d_prev)
    d_xt = xt_t.cuda()
    d_xn = torch.empty_like(d_xt)
    r = gc.make_recon(params["sampler"], a_t=params.get("a_t", 0), a_prev=params.get("a_prev", 0),
                      sigma=params.get("sigma", 0), sigma_next=params.get("sigma_next", 0))
    gc.transport_step(corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r, workspace=g.workspace(w.C),
                      update=update)
    torch.cuda.synchronize()
    gc.device_status()
    return (x0_prev, x0_new, xt64), d_out.cpu().numpy(), d_xn


def _check(w, got_x0, d_xn, ref_x0, ref_xn):
    assert_f32_close(got_x0, ref_x0, what="x0")
    if w.dtype == "bf16":
        assert_bf16_close(d_xn.cpu().view(torch.int16).numpy().view(np.uint16), ref_xn, what="x_next")
    else:
        assert_f32_close(d_xn.cpu().numpy(), ref_xn, scale=2.0, what="x_next")


@pytest.mark.parametrize("name", ["tiny", "hunyuan64", "solids96", "ring12_128"])
def test_value_copy_parity(gc, workloads, name):
    w = workloads(name)
    g = DeviceGeometry(w, K=w.K)
    anchors = oracle.rotate_anchors(w.N, w.a, 1)
    params = synth.recon_params(w, 2)
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    outs = {}
    for mode in ("sparse", "sparse_plain", "mask", "geometry", "table"):
        (x0_prev, x0_new, xt64), got, d_xn = _gpu_step(gc, w, g, g.corr_for(mode), anchors, params, "copy")
        ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=w.K,
                                                  geom=(w.pos, w.valid, w.cams, tau), x_t=xt64,
                                                  recon=recon_kw(params, None), update="copy")
        _check(w, got, d_xn, ref_x0, ref_xn)
        outs[mode] = got
    for mode in ("sparse_plain", "mask", "geometry", "table"):  # the same taps, weights and results
        np.testing.assert_array_equal(outs[mode], outs["sparse"])
    # the copy really differs from the delta transport on covered targets
    _, got_delta, _ = _gpu_step(gc, w, g, g.corr, anchors, params, "delta")
    non = [v for v in range(w.N) if v not in anchors]
    assert np.abs(outs["sparse"][:, non] - got_delta[:, non]).max() > 1e-2


def _pair_counts(g, w):
    T = g.gc.tiles_per_view(w.H, w.W)
    tp = g.tile_ptr.cpu().numpy().astype(np.int64)
    return tp[T::T] - tp[:-1:T]


@pytest.mark.parametrize("name", ["hunyuan64", "solids96", "batch128"])
def test_shuffled_correspondence_parity(gc, workloads, name):
    w = workloads(name)
    if name == "batch128":
        w = synth.make_workload("batch128", B=2)
    g = DeviceGeometry(w, K=w.K, tables=False)
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    idx, wt, _ = oracle.build_corr(w.pos, w.valid, w.cams, tau, K=w.K, with_band=False)
    counts = _pair_counts(g, w)
    # the records of each pair are the oracle's nonzero rows of that pair (both
    # sides decide in binary32, so this holds inside the threshold band too)
    np.testing.assert_array_equal(counts, (idx >= 0).any(-1).reshape(w.B * w.N * w.N, -1).sum(-1))
    perm = synth.pair_permutation(counts, seed=17)
    shuf = gc.permute_records(g.corr, torch.from_numpy(perm).cuda())
    anchors = oracle.rotate_anchors(w.N, w.a, 2)
    params = synth.recon_params(w, 4)
    (x0_prev, x0_new, xt64), got, d_xn = _gpu_step(gc, w, g, shuf, anchors, params)
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, table=oracle.shuffle_rows(idx, wt, perm),
                                              x_t=xt64, recon=recon_kw(params, None))
    _check(w, got, d_xn, ref_x0, ref_xn)
    # shuffling changes the result; the identity permutation does not
    _, base, _ = _gpu_step(gc, w, g, g.corr, anchors, params)
    assert np.abs(base - got).max() > 1e-3
    ident = gc.permute_records(g.corr, torch.arange(g.corr.c.max_records, dtype=torch.int32, device="cuda"))
    _, same, _ = _gpu_step(gc, w, g, ident, anchors, params)
    np.testing.assert_array_equal(same, base)
    # the shuffled records keep every target token and permute the taps
    rec0 = g.records.cpu().numpy()
    rec1 = shuf._keep["records"].cpu().numpy()
    np.testing.assert_array_equal(rec1[:, 0] & 0x0FFFFFFF, rec0[:, 0] & 0x0FFFFFFF)
    np.testing.assert_array_equal(rec1[:, 1:], rec0[perm, 1:])
    np.testing.assert_array_equal(rec1[:, 0] >> 28, rec0[perm, 0] >> 28)


def test_permutation_out_of_range_is_reported(gc, workloads):
    w = workloads("tiny")
    g = DeviceGeometry(w, K=4, tables=False)
    n = g.corr.c.max_records
    perm = torch.arange(n, dtype=torch.int32, device="cuda")
    perm[0] = n + 5  # bounds-checked in the kernel: the record is kept
    shuf = gc.permute_records(g.corr, perm)
    torch.cuda.synchronize()
    with pytest.raises(gc.GeocacheError) as ei:
        gc.device_status()
    assert ei.value.status == gc.EINVAL
    gc.device_status()  # cleared by the read
    np.testing.assert_array_equal(shuf._keep["records"].cpu().numpy(), g.records.cpu().numpy())


def test_shuffle_with_value_copy_interaction(gc, workloads):
    # Table 3's "shuf + value" cell: both ablations at once
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    idx, wt, _ = oracle.build_corr(w.pos, w.valid, w.cams, tau, K=4, with_band=False)
    perm = synth.pair_permutation(_pair_counts(g, w), seed=23)
    shuf = gc.permute_records(g.corr, torch.from_numpy(perm).cuda())
    anchors = oracle.rotate_anchors(w.N, w.a, 1)
    params = synth.recon_params(w, 6)
    (x0_prev, x0_new, xt64), got, d_xn = _gpu_step(gc, w, g, shuf, anchors, params, "copy")
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, table=oracle.shuffle_rows(idx, wt, perm),
                                              x_t=xt64, recon=recon_kw(params, None), update="copy")
    _check(w, got, d_xn, ref_x0, ref_xn)


@pytest.mark.parametrize("mode", ["sparse", "mask"])
def test_value_copy_in_place(gc, workloads, mode):
    # x0_out == x0_prev and x_next == x_t: the anchors' rows are written after
    # the gathers, covered targets are overwritten, the rest keep their state
    w = workloads("solids96")
    g = DeviceGeometry(w, K=w.K)
    anchors = oracle.rotate_anchors(w.N, w.a, 2)
    params = synth.recon_params(w, 3)
    x0_prev, x0_new, xt32 = step_inputs(w, 5, anchors)
    xt64, xt_t = latent_values(xt32, w)
    d_x0 = torch.from_numpy(x0_prev).cuda()
    d_new = torch.from_numpy(x0_new).cuda()
    d_x = xt_t.cuda()
    r = gc.make_recon(params["sampler"], a_t=params.get("a_t", 0), a_prev=params.get("a_prev", 0),
                      sigma=params.get("sigma", 0), sigma_next=params.get("sigma_next", 0))
    gc.transport_step(g.corr_for(mode), anchors, w.C, d_new, d_x0, d_x0, d_x, d_x, r, workspace=g.workspace(w.C),
                      update="copy")
    torch.cuda.synchronize()
    gc.device_status()
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=w.K, geom=(w.pos, w.valid, w.cams, tau),
                                              x_t=xt64, recon=recon_kw(params, None), update="copy")
    _check(w, d_x0.cpu().numpy(), d_x, ref_x0, ref_xn)
