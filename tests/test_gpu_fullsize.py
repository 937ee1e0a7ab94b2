"""Parity at the benchmark's full size and launch configuration: the batch128
workload at 128 assets (the bench's default: the largest point of the workload's batch
sweep), sparse mode, bf16 latents and an f32 cache, one cached DDIM step, on
outputs the oracle computes one by one: tau for every asset, the keep masks
of sampled (target, source, token) rows, and x0(t) / x_{t-1} at a sample of
target pixels of every view (Eq. 1 with the multi-anchor aggregation and the
closed-form DDIM conversion of Sec. 3.2).  The delta transport and the
value-copy ablation (Sec. 4.3) are both checked."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_13255_gb300 import synth

from gpu_helpers import DeviceGeometry, assert_bf16_close, assert_f32_close, latent_values, recon_kw, step_inputs

pytestmark = pytest.mark.gpu

B_BENCH = 128


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13255_gb300 import build as gbuild
    gbuild.build()
    from paper_2608_13255_gb300 import geocache
    geocache.load()
    return geocache


@pytest.fixture(scope="module")
def full(gc):
    w = synth.make_workload("batch128", B=B_BENCH)
    return w, DeviceGeometry(w, K=4, tables=False)


def test_tau_and_sampled_keep_masks(gc, full):
    w, g = full
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    np.testing.assert_array_equal(g.tau.cpu().numpy(), tau)
    keep = g.keep.cpu().numpy()
    rng = np.random.default_rng(5)
    n, hits = 4096, 0
    fg = np.argwhere(w.valid > 0)  # sample foreground targets: background rows are trivially zero
    pick = fg[rng.integers(0, len(fg), n)]
    for k in range(n):
        bb, vv, jj, ii = pick[k]
        uu = (vv + 1 + k % (w.N - 1)) % w.N
        X = w.pos[bb, vv, jj, ii]
        idx, _ = oracle.taps(w.cams[bb, uu], w.pos[bb, uu], w.valid[bb, uu], X, tau[bb], K=4)
        mask = sum(1 << t for t in range(4) if idx[t] >= 0)
        assert keep[bb, vv, uu, jj, ii] == mask, (bb, vv, uu, jj, ii)
        hits += mask != 0
    assert hits > n // 50  # the sample reaches kept rows


@pytest.mark.parametrize("update", ["delta", "copy"])
def test_cached_step_sampled_pixels(gc, full, update):
    w, g = full
    anchors = oracle.rotate_anchors(w.N, w.a, 1)
    params = synth.recon_params(w, 1)
    x0_prev, x0_new, xt32 = step_inputs(w, 1, anchors)
    xt64, xt_t = latent_values(xt32, w)
    d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
    d_out = torch.empty_like(d_prev)
    d_xt = xt_t.cuda()
    d_xn = torch.empty_like(d_xt)
    r = gc.make_recon(params["sampler"], a_t=params.get("a_t", 0), a_prev=params.get("a_prev", 0))
    gc.transport_step(g.corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r, workspace=g.workspace(w.C),
                      update=update)
    torch.cuda.synchronize()
    gc.device_status()
    # 1% of the target pixels of every view, plus every covered pixel of one asset's views
    rng = np.random.default_rng(9)
    sel = (rng.random((w.B, w.N, w.H * w.W)) < 0.01).astype(np.uint8)
    sel[3] = 1
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=4, geom=(w.pos, w.valid, w.cams, tau),
                                              x_t=xt64, recon=recon_kw(params, None), sel=sel, update=update)
    m = np.broadcast_to(sel.reshape(w.B, w.N, 1, w.H, w.W) > 0, x0_prev.shape)
    got = d_out.cpu().numpy()
    assert_f32_close(got[m], ref_x0[m], what="x0 (sampled)")
    bits = d_xn.cpu().view(torch.int16).numpy().view(np.uint16)
    assert_bf16_close(bits[m], ref_xn[m], what="x_next (sampled)")
    non = [v for v in range(w.N) if v not in anchors]
    moved = np.abs(ref_x0[3, non] - x0_prev[3, non]).max()
    assert moved > 1e-3  # the sample contains transported targets


def test_ring12_x8_cached_step_sampled_pixels(gc):
    # the bench's 12-view leg in its launch configuration: ring12_128 (12
    # views, 128 x 128 x 16 bf16 latents, 4 anchors, FM-Euler) replicated to
    # 8 assets, no source index and the workspace the bench allocates, so
    # the step takes the increment-plane path; every anchor set of the
    # rotation, x0(t) and x_{t-1} at 1% of the target pixels plus every
    # pixel of one asset against the oracle
    w = synth.replicate_assets(synth.make_workload("ring12_128"), 8)
    g = DeviceGeometry(w, K=4, tables=False, source_index=False)
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    rng = np.random.default_rng(12)
    sel = (rng.random((w.B, w.N, w.H * w.W)) < 0.01).astype(np.uint8)
    sel[5] = 1
    m = None
    for ordinal in range(3):  # the strided rotation of 4 anchors among 12 views has 3 sets
        anchors = oracle.rotate_anchors(w.N, w.a, ordinal)
        params = synth.recon_params(w, 2 + ordinal)
        x0_prev, x0_new, xt32 = step_inputs(w, 2 + ordinal, anchors)
        xt64, xt_t = latent_values(xt32, w)
        d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
        d_out = torch.empty_like(d_prev)
        d_xt = xt_t.cuda()
        d_xn = torch.empty_like(d_xt)
        r = gc.make_recon(params["sampler"], sigma=params["sigma"], sigma_next=params["sigma_next"])
        gc.transport_step(g.corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r, workspace=g.workspace(w.C))
        torch.cuda.synchronize()
        gc.device_status()
        ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=4,
                                                  geom=(w.pos, w.valid, w.cams, tau), x_t=xt64,
                                                  recon=recon_kw(params, None), sel=sel)
        if m is None:
            m = np.broadcast_to(sel.reshape(w.B, w.N, 1, w.H, w.W) > 0, x0_prev.shape)
        assert_f32_close(d_out.cpu().numpy()[m], ref_x0[m], what="x0 (sampled, anchors %s)" % anchors)
        bits = d_xn.cpu().view(torch.int16).numpy().view(np.uint16)
        assert_bf16_close(bits[m], ref_xn[m], what="x_next (sampled, anchors %s)" % anchors)
        non = [v for v in range(w.N) if v not in anchors]
        assert np.abs(ref_x0[5, non] - x0_prev[5, non]).max() > 1e-3
