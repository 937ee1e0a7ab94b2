"""Failure handling on the GPU without a fault: a bounded wait inside the
staged transport kernel is made to run out (its first unit's copies are
never issued, through the geocache_debug_set_wait test hook), the kernel
reports it in the device status word instead of hanging or trapping, the
host reads GEOCACHE_ETIMEOUT, and the next call on the same context is
correct."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_13255_gb300 import synth

from gpu_helpers import DeviceGeometry, assert_bf16_close, assert_f32_close, latent_values, recon_kw, step_inputs

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


def _inputs(w, anchors):
    x0_prev, x0_new, xt32 = step_inputs(w, 3, anchors)
    xt64, xt = latent_values(xt32, w)
    return x0_prev, x0_new, xt64, xt


def test_wait_that_runs_out_is_reported_and_the_context_stays_usable(gc, workloads):
    w = workloads("hunyuan64")  # 64 x 64 tokens: rows suit the staged (bulk-copy) kernel
    g = DeviceGeometry(w, K=4, tables=False)
    corr = g.corr_for("mask")
    anchors = [0, 3]
    x0_prev, x0_new, xt64, xt = _inputs(w, anchors)
    p = synth.recon_params(w, 4)
    r = gc.make_recon("ddim", a_t=p["a_t"], a_prev=p["a_prev"])
    d_prev, d_new, d_xt = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda(), xt.cuda()
    gc.device_status()  # nothing pending
    sentinel = float("nan")
    out = torch.full_like(d_prev, sentinel)
    xn = torch.empty_like(d_xt)
    gc.debug_set_wait(200_000, drop_first_copy=True)  # 200 us limit; unit 0's copies are never issued
    try:
        gc.transport_step(corr, anchors, w.C, d_new, d_prev, out, d_xt, xn, r)
        torch.cuda.synchronize()  # the kernel ended: the wait gave up instead of hanging
        with pytest.raises(gc.GeocacheError) as ei:
            gc.device_status()
        assert ei.value.status == gc.ETIMEOUT
        gc.device_status()  # the read cleared the word
    finally:
        gc.debug_set_wait(0, drop_first_copy=False)
    # the CTA that gave up wrote nothing: with one unit per CTA at this size,
    # unit 0 (asset 0, view 0, first 1024 tokens, channels 0-3) keeps the
    # sentinel and every other unit holds its result
    tau = oracle.tau(w.pos, w.valid, w.tol_frac)
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=4, geom=(w.pos, w.valid, w.cams, tau),
                                              x_t=xt64, recon=recon_kw(p))
    got = out.cpu().numpy()
    unit0 = np.zeros(got.shape, bool)
    unit0[0, 0, 0:4].reshape(4, -1)[:, :1024] = True
    assert np.isnan(got[unit0]).all()
    assert_f32_close(got[~unit0], ref_x0[~unit0], what="x0 outside the unit that gave up")
    # the next call on the same context is complete and correct
    out2, xn2 = torch.empty_like(d_prev), torch.empty_like(d_xt)
    gc.transport_step(corr, anchors, w.C, d_new, d_prev, out2, d_xt, xn2, r)
    torch.cuda.synchronize()
    gc.device_status()
    assert_f32_close(out2.cpu().numpy(), ref_x0, what="x0 after the timeout")
    assert_bf16_close(xn2.cpu().view(torch.int16).numpy().view(np.uint16), ref_xn, what="x_next after the timeout")


def test_wait_limit_restored_by_default(gc, workloads):
    # a short limit that every copy meets: no timeout is reported
    w = workloads("hunyuan64")
    g = DeviceGeometry(w, K=4, tables=False)
    anchors = [1, 4]
    x0_prev, x0_new, _, _ = _inputs(w, anchors)
    d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
    gc.debug_set_wait(100_000_000)  # 100 ms
    try:
        out = torch.empty_like(d_prev)
        gc.transport_step(g.corr_for("mask"), anchors, w.C, d_new, d_prev, out)
        torch.cuda.synchronize()
        gc.device_status()
    finally:
        gc.debug_set_wait(0)
    assert torch.isfinite(out).all()
