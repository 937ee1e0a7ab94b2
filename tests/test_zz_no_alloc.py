"""The cached step without a caller-provided workspace
(geocache_transport_step_noalloc), for callers that cannot allocate device
memory where they run a step: its results must equal the regular entry
point's bit for bit on consecutive calls (both run the same kernels on the
same inputs, so any difference would be stale or shared scratch), and steps
needing more scratch than the built-in array holds must be rejected before
anything runs.

The file name makes pytest collect it last."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_13255_gb300 import synth

from gpu_helpers import DeviceGeometry, latent_values, step_inputs

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


def _step(gc, g, w, anchors, step, noalloc, in_place):
    x0_prev, x0_new, xt32 = step_inputs(w, step, anchors)
    _, xt = latent_values(xt32, w)
    d_prev, d_new, d_xt = (torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda(), xt.cuda())
    d_out = d_prev if in_place else torch.empty_like(d_prev)
    d_xn = d_xt if in_place else torch.empty_like(d_xt)
    p = synth.recon_params(w, step)
    r = gc.make_recon(p["sampler"], a_t=p.get("a_t", 0), a_prev=p.get("a_prev", 0), sigma=p.get("sigma", 0),
                      sigma_next=p.get("sigma_next", 0))
    if noalloc:
        gc.transport_step_noalloc(g.corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r)
    else:
        gc.transport_step(g.corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r, workspace=g.workspace(w.C))
    torch.cuda.synchronize()
    gc.device_status()
    return d_out.cpu(), d_xn.cpu(), x0_prev


@pytest.mark.parametrize("in_place", [False, True])
@pytest.mark.parametrize("sampler,lat", [("ddim", "bf16"), ("fm_euler", "bf16"), ("ddim", "f32")])
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(gc, sampler, lat, in_place):
    w = synth.make_workload("batch128", B=2)
    w = synth.Workload(**{**w.__dict__, "sampler": sampler, "dtype": lat, "S": 30})
    g = DeviceGeometry(w, K=4, tables=False)
    assert 0 < g.corr.workspace_floats(w.C) <= 4 * 1024 * 1024
    # two calls in a row with different anchors and inputs: the second call
    # starts from the scratch the first one left behind
    for anchors, step in (([0, 3], 1), ([1, 4], 2)):
        ref_x0, ref_xn, _ = _step(gc, g, w, anchors, step, noalloc=False, in_place=in_place)
        got_x0, got_xn, x0_prev = _step(gc, g, w, anchors, step, noalloc=True, in_place=in_place)
        assert torch.equal(got_x0.view(torch.int32), ref_x0.view(torch.int32)), "x0 differs (no-alloc vs workspace)"
        bits = torch.int16 if lat == "bf16" else torch.int32
        assert torch.equal(got_xn.view(bits), ref_xn.view(bits)), "x_next differs (no-alloc vs workspace)"
        # the step really transported something
        assert np.abs(got_x0.numpy() - x0_prev).max() > 1e-3


def test_noalloc_wide_latents_match_the_plane_path(gc):
    # ring12_128 (C = 16): the built-in array holds max_records * C floats but
    # not the anchors' increment plane as well, so the no-alloc step applies
    # the records into rows while the workspace entry point (sized by
    # geocache_transport_workspace) takes the plane; the bits must agree
    w = synth.make_workload("ring12_128")
    g = DeviceGeometry(w, K=4, tables=False, source_index=False)
    need = g.corr.min_workspace_floats(w.C)
    plane = w.B * w.a * 4 * (-(-w.C // 4)) * w.H * w.W
    assert need <= 4 * 1024 * 1024 < need + plane
    for anchors, step in (([0, 3, 6, 9], 2), ([1, 4, 7, 10], 3)):
        for in_place in (False, True):
            ref_x0, ref_xn, _ = _step(gc, g, w, anchors, step, noalloc=False, in_place=in_place)
            got_x0, got_xn, _ = _step(gc, g, w, anchors, step, noalloc=True, in_place=in_place)
            assert torch.equal(got_x0.view(torch.int32), ref_x0.view(torch.int32))
            assert torch.equal(got_xn.view(torch.int16), ref_xn.view(torch.int16))


def test_noalloc_rejects_steps_beyond_its_scratch(gc):
    # a sparse-mode step whose scratch (max_records * C floats) exceeds the
    # built-in array is refused before any launch
    c = gc.Corr(1, 6, 8, 8, 4, 0.01, 16, 16, 16, 16, None, None, 16, 16, 16, 2 * 1024 * 1024, gc.CORR_SPARSE)
    anc = (ctypes.c_int32 * 2)(0, 3)
    st = gc.load().geocache_transport_step_noalloc(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16,
                                                   32, None, None, 0, None, None)
    assert st == gc.ESHAPE
    assert "scratch" in gc.last_error()


def test_noalloc_accepts_a_full_anchor_step_of_a_large_corr(gc):
    # with every view an anchor no record is applied, so no scratch is needed
    # however large the sparse form is: the step runs and equals the
    # denoiser's x0 (a = N)
    w = synth.make_workload("batch128", B=1)
    g = DeviceGeometry(w, K=4, tables=False)
    big = gc.Corr.from_buffer_copy(g.corr.c)
    big.max_records = 64 * 1024 * 1024  # larger than the built-in array at C = 4 (the records are not read)
    handle = gc.CorrHandle(big, g.corr._keep)
    anchors = list(range(w.N))
    x0_prev, x0_new, _ = step_inputs(w, 1, anchors)
    d_prev, d_new = torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda()
    out = torch.empty_like(d_prev)
    gc.transport_step_noalloc(handle, anchors, w.C, d_new, d_prev, out)
    torch.cuda.synchronize()
    gc.device_status()
    assert torch.equal(out, d_new)
