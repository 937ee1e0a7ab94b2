"""The cached step without a caller-provided workspace
(geocache_transport_step_noalloc), for callers that cannot allocate device
memory where they run a step: its results must equal the regular entry
point's on consecutive calls, and steps needing more scratch than the
built-in array holds must be rejected before anything runs.

The file name makes pytest collect it last."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2608_13255_gb300 import synth

from gpu_helpers import DeviceGeometry, assert_bf16_close, assert_f32_close, bf16_to_f64, latent_values, step_inputs

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


def _step(gc, g, w, anchors, step, noalloc):
    x0_prev, x0_new, xt32 = step_inputs(w, step, anchors)
    _, xt = latent_values(xt32, w)
    d_prev, d_new, d_xt = (torch.from_numpy(x0_prev).cuda(), torch.from_numpy(x0_new).cuda(), xt.cuda())
    d_out, d_xn = torch.empty_like(d_prev), torch.empty_like(d_xt)
    p = synth.recon_params(w, step)
    r = gc.make_recon("ddim", a_t=p["a_t"], a_prev=p["a_prev"])
    if noalloc:
        gc.transport_step_noalloc(g.corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r)
    else:
        gc.transport_step(g.corr, anchors, w.C, d_new, d_prev, d_out, d_xt, d_xn, r, workspace=g.workspace(w.C))
    torch.cuda.synchronize()
    return d_out.cpu().numpy(), d_xn.cpu().view(torch.int16).numpy().view(np.uint16)


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(gc):
    w = synth.make_workload("batch128", B=2)
    g = DeviceGeometry(w, K=4, tables=False)
    assert 0 < g.corr.workspace_floats(w.C) <= 4 * 1024 * 1024
    # two calls in a row with different anchors and inputs: the second call
    # starts from the scratch the first one left behind
    for anchors, step in (([0, 3], 1), ([1, 4], 2)):
        ref_x0, ref_xn = _step(gc, g, w, anchors, step, noalloc=False)
        got_x0, got_xn = _step(gc, g, w, anchors, step, noalloc=True)
        assert_f32_close(got_x0, ref_x0, what="x0 (no-alloc vs workspace)")
        assert_bf16_close(got_xn, bf16_to_f64(ref_xn), what="x_next (no-alloc vs workspace)")
        # the step really transported something
        x0_prev = step_inputs(w, step, anchors)[0]
        assert np.abs(got_x0 - x0_prev).max() > 1e-3


def test_noalloc_rejects_steps_beyond_its_scratch(gc):
    # a sparse-mode step whose scratch (max_records * C floats) exceeds the
    # built-in array is refused before any launch
    c = gc.Corr(1, 6, 8, 8, 4, 0.01, 16, 16, 16, 16, None, None, 16, 16, 16, 2 * 1024 * 1024, gc.CORR_SPARSE)
    anc = (ctypes.c_int32 * 2)(0, 3)
    st = gc.load().geocache_transport_step_noalloc(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16,
                                                   32, None, None, 0, None, None)
    assert st == gc.ESHAPE
    assert "scratch" in gc.last_error()
