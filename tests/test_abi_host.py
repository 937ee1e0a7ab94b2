"""Host-side checks of the C ABI (no GPU needed): the library builds and
loads, exports every entry point that include/geocache.h declares, and its
host logic (refresh schedule, anchor rotation, argument checking) behaves as
documented.  Rotation and schedule are compared with the oracle's
independent implementation (Sec. 3.2, batch-sliced anchor forward and
drift-bounding schedule)."""
import ctypes
import os
import re

import pytest

import oracle
from paper_2608_13255_gb300 import build as gbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def gc():
    gbuild.build()
    from paper_2608_13255_gb300 import geocache
    geocache.load()
    return geocache


def _declared():
    src = open(os.path.join(ROOT, "include", "geocache.h")).read()
    return sorted(set(re.findall(r"^(?:int|const char\*)\s+(geocache_\w+)\s*\(", src, re.M)))


def test_exports_every_declared_symbol(gc):
    names = _declared()
    assert len(names) >= 7
    L = gc.load()
    for n in names:
        assert hasattr(L, n), n
    assert gc.abi_version() == 2


SCHEDS = [
    {"kind": "every_k", "k": 5},
    {"kind": "every_k", "k": 4},
    {"kind": "head_mid_tail", "head": 2, "mid": 1, "tail": 1},
    {"kind": "head_mid_tail", "head": 2, "mid": 0, "tail": 1},
    {"kind": "list", "steps": [0, 3, 7]},
    {"kind": "all_full"},
    {"kind": "single_cached"},
]


@pytest.mark.parametrize("sched", SCHEDS, ids=lambda s: s["kind"] + str(s.get("k", s.get("mid", ""))))
def test_schedule_matches_oracle(gc, sched):
    for S in (1, 10, 30, 50):
        for t in range(S):
            assert gc.is_full_step(t, S, sched) == oracle.is_full_step(t, S, sched), (t, S)


@pytest.mark.parametrize("N,a", [(6, 2), (6, 3), (12, 4), (10, 2), (6, 4), (7, 3), (6, 6), (6, 1)])
def test_rotation_matches_oracle(gc, N, a):
    sched = {"kind": "every_k", "k": 5}
    S = 30
    for t in range(S):
        anchors, full = gc.rotate_anchors(N, a, t, S, sched)
        assert full == oracle.is_full_step(t, S, sched)
        assert anchors == oracle.rotate_anchors(N, a, oracle.cached_ordinal(t, S, sched))
    contig = dict(sched, contiguous=1)
    for t in range(S):
        anchors, _ = gc.rotate_anchors(N, a, t, S, contig)
        assert anchors == oracle.rotate_anchors(N, a, oracle.cached_ordinal(t, S, sched), contiguous=True)


def test_tiny_first_cached_step_anchors(gc):
    assert gc.rotate_anchors(6, 2, 1, 1 + 1, {"kind": "single_cached"}) == ([0, 3], False)


def test_argument_errors_before_launch(gc):
    L = gc.load()
    # NULL corr, bad sizes, bad anchors, bad sampler: rejected on the host
    assert L.geocache_transport_step(None, None, 0, 0, None, None, None, None, None, 0, None, None, 0, None) == gc.EINVAL
    assert "corr" in gc.last_error()
    c = gc.Corr(1, 6, 8, 8, 4, 0.01, 16, 16, 16, 16, None, None, None, gc.CORR_GEOMETRY)
    anc = (ctypes.c_int32 * 2)(3, 0)  # not ascending
    st = L.geocache_transport_step(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16, 32,
                                   None, None, 0, None, None, 0, None)
    assert st == gc.EINVAL and "ascending" in gc.last_error()
    anc = (ctypes.c_int32 * 2)(0, 3)
    st = L.geocache_transport_step(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 0, 16, 16, 32,
                                   None, None, 0, None, None, 0, None)
    assert st == gc.ESHAPE
    c.K = 3
    st = L.geocache_transport_step(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16, 32,
                                   None, None, 0, None, None, 0, None)
    assert st == gc.EINVAL
    c.K = 4
    c.mode = gc.CORR_MASK  # mask mode without keep masks
    st = L.geocache_transport_step(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16, 32,
                                   None, None, 0, None, None, 0, None)
    assert st == gc.EINVAL and "keep" in gc.last_error()
    c.mode = gc.CORR_SPARSE  # sparse mode without records / workspace
    st = L.geocache_transport_step(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16, 32,
                                   None, None, 0, None, None, 0, None)
    assert st == gc.EINVAL and "tile_ptr" in gc.last_error()
    c.tile_ptr, c.records, c.max_records = 64, 128, 10
    st = L.geocache_transport_step(ctypes.byref(c), ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16, 32,
                                   None, None, 0, None, None, 0, None)
    assert st == gc.EINVAL and "workspace" in gc.last_error()
    assert L.geocache_transport_workspace(ctypes.byref(c), 4) == 40
    c.tile_ptr, c.records, c.max_records = None, None, 0
    c.mode = gc.CORR_GEOMETRY
    assert L.geocache_transport_workspace(ctypes.byref(c), 4) == 0
    c.N = 65
    assert L.geocache_build_corr(ctypes.byref(c), None) == gc.ESHAPE
    c.N = 6
    r = gc.make_recon("ddim", a_t=1.0, a_prev=0.5)
    st = L.geocache_reconstruct(16, 16, 32, 1, 10, ctypes.byref(r), None, None)
    assert st == gc.EINVAL and "a_t" in gc.last_error()
    r = gc.make_recon("fm_euler", sigma=0.5, sigma_next=0.4, pred_kind="eps")
    st = L.geocache_reconstruct(16, 16, 32, 1, 10, ctypes.byref(r), None, None)
    assert st == gc.EINVAL
    r = gc.make_recon("ddim", a_t=0.5, a_prev=0.6)
    assert L.geocache_reconstruct(16, 16, 32, 7, 10, ctypes.byref(r), None, None) == gc.EDTYPE
    assert L.geocache_reconstruct(16, 16, 32, 1, -1, ctypes.byref(r), None, None) == gc.ESHAPE
    # partial overlap of x_next and x_t (bf16, 10 elements = 20 bytes)
    assert L.geocache_reconstruct(1000, 4096, 1010, 1, 10, ctypes.byref(r), None, None) == gc.EALIAS
    # schedule / rotation argument errors
    s, _k = gc.make_schedule({"kind": "every_k", "k": 0})
    assert L.geocache_is_full_step(3, 10, ctypes.byref(s)) == gc.EINVAL
    assert L.geocache_is_full_step(10, 10, ctypes.byref(s)) == gc.ESHAPE
    out = (ctypes.c_int32 * 8)()
    s, _k = gc.make_schedule({"kind": "every_k", "k": 5})
    assert L.geocache_rotate_anchors(6, 7, 1, 10, ctypes.byref(s), ctypes.cast(out, ctypes.c_void_p), None) == gc.EINVAL
    assert gc.last_error() != ""


def test_ablation_entry_points_check_arguments(gc):
    L = gc.load()
    c = gc.Corr(1, 6, 8, 8, 4, 0.01, 16, 16, 16, 16, None, None, None, None, None, 0, gc.CORR_SPARSE)
    anc = (ctypes.c_int32 * 2)(0, 3)
    st = L.geocache_transport_step_update(ctypes.byref(c), 7, ctypes.cast(anc, ctypes.c_void_p), 2, 4, 16, 16, 32,
                                          None, None, 0, None, None, 0, None)
    assert st == gc.EINVAL and "update" in gc.last_error()
    # the permutation needs records, a permutation and an output
    assert L.geocache_permute_records(None, 16, 32, None) == gc.EINVAL
    assert L.geocache_permute_records(ctypes.byref(c), 16, 32, None) == gc.EINVAL
    assert "records" in gc.last_error()
    c.records, c.max_records = 4096, 64
    assert L.geocache_permute_records(ctypes.byref(c), 16, 4096 + 512, None) == gc.EALIAS  # out overlaps records
    assert L.geocache_permute_records(ctypes.byref(c), 16, 4100, None) == gc.EINVAL  # misaligned out


def test_raster_entry_point_checks_arguments(gc):
    L = gc.load()
    P = 4096
    # sizes
    assert L.geocache_raster_posmaps(P, 3, P, 1, P, 0, P, 6, 8, 8, P, P, P, None) == gc.ESHAPE
    assert L.geocache_raster_posmaps(P, 3, P, 1, P, 1, P, 65, 8, 8, P, P, P, None) == gc.ESHAPE
    assert L.geocache_raster_posmaps(P, -1, P, 1, P, 1, P, 6, 8, 8, P, P, P, None) == gc.ESHAPE
    # required buffers, alignment, overlaps
    assert L.geocache_raster_posmaps(None, 3, P, 1, P, 1, P, 6, 8, 8, P, P, P, None) == gc.EINVAL
    assert L.geocache_raster_posmaps(P, 3, P, 1, P, 1, P, 6, 8, 8, P + 4, 1 << 20, 1 << 21, None) == gc.EINVAL
    st = L.geocache_raster_posmaps(1 << 24, 3, 1 << 25, 1, 1 << 26, 1, 1 << 27, 6, 8, 8, 1 << 20, 1 << 20, 1 << 22, None)
    assert st == gc.EALIAS and "overlap" in gc.last_error()
    st = L.geocache_raster_posmaps(1 << 20, 3, 1 << 25, 1, 1 << 26, 1, 1 << 27, 6, 8, 8, 1 << 20, 1 << 21, 1 << 22, None)
    assert st == gc.EALIAS  # zbuf over the vertices
