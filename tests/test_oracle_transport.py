"""Pins of the oracle's delta transport, reconstruction, bf16 rounding and
schedule (Eq. 1 and the surrounding paragraphs of Sec. 3.2; Table 1).

The checks are chosen so that a plausible slip in the oracle (a dropped term,
a wrong sign, a swapped anchor/target index, a transposed operand, a missing
division by the number of covering anchors) fails at least one of them.
"""
import math
import os

import numpy as np
import pytest

import oracle
from paper_2608_13255_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _setup(w, anchors, seed=0, std=0.1):
    rng = np.random.default_rng(seed)
    shp = (w.B, w.N, w.C, w.H, w.W)
    x0_prev = rng.standard_normal(shp)
    x0_new = x0_prev[:, anchors] + std * rng.standard_normal((w.B, len(anchors), w.C, w.H, w.W))
    return x0_prev, x0_new


def _dense_operator(w, tau, u, v, K):
    """G_{u->v} as a dense [HW, HW] matrix assembled from brute-force rows."""
    HW = w.H * w.W
    G = np.zeros((HW, HW))
    for p in np.flatnonzero(w.valid[0, v].reshape(-1)):
        X = w.pos[0, v].reshape(-1, 3)[p]
        for q, x in oracle.brute_row(w.cams[0, u], w.pos[0, u], w.valid[0, u], X, tau, K=K):
            G[p, q] = x
    return G


@pytest.mark.parametrize("K", [4, 1])
def test_transport_matches_dense_brute_force_operator(K):
    # Eq. 1 with the normalised multi-anchor sum, written as dense linear
    # algebra on operators assembled from the brute-force rows
    w = synth.make_workload("hunyuan64", H=16, W=16)
    anchors = [1, 4]
    # a tolerance of about one token at 16x16 so that many targets are covered
    tau = np.float32([0.12])
    x0_prev, x0_new = _setup(w, anchors)
    x0_out, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=K,
                                         geom=(w.pos, w.valid, w.cams, tau))
    max_cover = 0
    for v in range(w.N):
        if v in anchors:
            np.testing.assert_array_equal(x0_out[0, v], x0_new[0, anchors.index(v)])
            continue
        Gs = [_dense_operator(w, tau[0], u, v, K) for u in anchors]
        cover = sum((G.sum(1) > 0).astype(float) for G in Gs)  # n per target pixel
        max_cover = max(max_cover, cover.max())
        for c in range(w.C):
            inc = sum(G @ (x0_new[0, s, c].reshape(-1) - x0_prev[0, u, c].reshape(-1))
                      for s, (u, G) in enumerate(zip(anchors, Gs)))
            ref = x0_prev[0, v, c].reshape(-1) + np.where(cover > 0, inc / np.maximum(cover, 1), 0.0)
            # rows differing only by taps with weight below 1e-6 (rounding of
            # the footprint fraction) agree to ~1e-6 of the increment
            np.testing.assert_allclose(x0_out[0, v, c].reshape(-1), ref, atol=2e-6, rtol=0)
    assert max_cover == 2  # some target is covered by both anchors


def test_identity_camera_reproduces_anchor_delta():
    # target camera equal to the anchor camera: x0^v(t) - x0^v(t-1) = delta^u
    # at every foreground pixel (exact for K=1, to rounding for K=4)
    w = synth.make_workload("hunyuan64", H=32, W=32)
    w.cams[0, 1] = w.cams[0, 0]
    w.pos[0, 1], w.valid[0, 1] = w.pos[0, 0], w.valid[0, 0]
    tau = oracle.tau(w.pos, w.valid)
    anchors = [0]
    x0_prev, x0_new = _setup(w, anchors, seed=3)
    d0 = x0_new[0, 0] - x0_prev[0, 0]
    fg = w.valid[0, 1] > 0
    for K, tol in ((1, 1e-15), (4, 1e-5)):
        x0_out, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=K, geom=(w.pos, w.valid, w.cams, tau))
        got = (x0_out[0, 1] - x0_prev[0, 1])[:, fg]
        np.testing.assert_allclose(got, d0[:, fg], atol=tol * 4, rtol=0)
        # background keeps its state exactly (invalid-match rule)
        np.testing.assert_array_equal(x0_out[0, 1][:, ~fg], x0_prev[0, 1][:, ~fg])


def test_exact_centre_projections_keep_one_tap_and_reproduce_the_delta():
    # a camera-aligned plane whose positions project exactly onto the token
    # centres, seen by two identical cameras: every footprint fraction is
    # exactly 0, so the zero-weight rule leaves the single tap at the target's
    # own token with weight 1 (K = 4 and K = 1 alike), and the target's x0
    # changes by exactly the anchor's delta (Sec. 3.2, correspondence operator
    # and Eq. 1 with one covering anchor)
    w = synth.identity_camera_pair(synth.make_workload("hunyuan64", H=32, W=32), plane=True)
    tau = oracle.tau(w.pos, w.valid)
    fg = w.valid[0, 1].reshape(-1) > 0
    p = np.flatnonzero(fg)
    # the closed form of the projection: token (i, j) lands on (i + 0.5, j + 0.5)
    cam = w.cams[0, 0]
    for q in p[:: max(1, len(p) // 50)]:
        uu, vv = oracle.project(cam, w.pos[0, 0].reshape(-1, 3)[q])[:2]
        assert (uu, vv) == (q % w.W + 0.5, q // w.W + 0.5)
    anchors = [0]
    x0_prev, x0_new = _setup(w, anchors, seed=5)
    d0 = x0_new[0, 0] - x0_prev[0, 0]
    for K in (4, 1):
        idx, wt, band = oracle.build_corr(w.pos, w.valid, w.cams, tau, K=K)
        assert band.sum() == 0
        row, wrow = idx[0, 1, 0].reshape(-1, K), wt[0, 1, 0].reshape(-1, K)
        np.testing.assert_array_equal(row[fg, 0], p)
        assert (wrow[fg, 0] == 1.0).all()
        assert (row[fg, 1:] == -1).all() and (wrow[fg, 1:] == 0.0).all()
        assert (row[~fg] == -1).all()
        x0_out, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=K, geom=(w.pos, w.valid, w.cams, tau))
        got = (x0_out[0, 1] - x0_prev[0, 1]).reshape(w.C, -1)
        np.testing.assert_allclose(got[:, fg], d0.reshape(w.C, -1)[:, fg], atol=1e-12, rtol=0)
        np.testing.assert_array_equal(got[:, ~fg], 0.0)


def test_zero_delta_leaves_targets_unchanged(workloads):
    w = workloads("hunyuan64")
    anchors = [0, 3]
    tau = oracle.tau(w.pos, w.valid)
    x0_prev, _ = _setup(w, anchors)
    x0_new = x0_prev[:, anchors].copy()
    x0_out, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, geom=(w.pos, w.valid, w.cams, tau))
    np.testing.assert_array_equal(x0_out, x0_prev)


def test_transport_is_linear_and_convex(workloads):
    w = workloads("hunyuan64")
    anchors = [1, 4]
    tau = oracle.tau(w.pos, w.valid)
    table = oracle.build_corr(w.pos, w.valid, w.cams, tau)[:2]
    rng = np.random.default_rng(7)
    shp = (w.B, len(anchors), w.C, w.H, w.W)
    base = rng.standard_normal((w.B, w.N, w.C, w.H, w.W))
    d1, d2 = rng.standard_normal(shp), rng.standard_normal(shp)
    zero = np.zeros_like(base)

    def T(d):  # transported increment with a zero previous state
        return oracle.transport_step(anchors, d, zero, table=table)[0]

    al, be = 0.7, -1.3
    lhs = T(al * d1 + be * d2)
    rhs = al * T(d1) + be * T(d2)
    non = [v for v in range(w.N) if v not in anchors]
    np.testing.assert_allclose(lhs[:, non], rhs[:, non], atol=1e-12)
    # convexity: no target increment exceeds the largest anchor increment
    g = np.abs(T(d1)[:, non]).max()
    assert g <= np.abs(d1).max() + 1e-12
    # the increment is independent of the target's own previous state
    out_a = oracle.transport_step(anchors, d1 + base[:, anchors], base, table=table)[0]
    np.testing.assert_allclose((out_a - base)[:, non], T(d1)[:, non], atol=1e-12)


def test_table_and_geometry_paths_agree(workloads):
    w = workloads("solids96")
    anchors = [0, 2, 4]
    tau = oracle.tau(w.pos, w.valid)
    x0_prev, x0_new = _setup(w, anchors)
    table = oracle.build_corr(w.pos, w.valid, w.cams, tau)[:2]
    a = oracle.transport_step(anchors, x0_new, x0_prev, table=table)[0]
    b = oracle.transport_step(anchors, x0_new, x0_prev, geom=(w.pos, w.valid, w.cams, tau))[0]
    np.testing.assert_array_equal(a, b)


# ------------------------------------------------------- reconstruction --
def test_ddim_round_trip_and_v():
    rng = np.random.default_rng(1)
    x0 = rng.standard_normal(1000)
    eps0 = rng.standard_normal(1000)
    for ab in (0.02, 0.5, 0.97):
        xt = math.sqrt(ab) * x0 + math.sqrt(1 - ab) * eps0
        # a step to the same noise level returns x_t; eps is recovered
        xn, eps = oracle.reconstruct(xt, x0, oracle.DDIM, a_t=ab, a_prev=ab, pred_kind=oracle.PRED_EPS)
        np.testing.assert_allclose(eps, eps0, atol=1e-12 / math.sqrt(1 - ab))
        np.testing.assert_allclose(xn, xt, atol=1e-13)
        # v-prediction: x0 = sqrt(ab) x_t - sqrt(1-ab) v (standard identity)
        _, v = oracle.reconstruct(xt, x0, oracle.DDIM, a_t=ab, a_prev=ab, pred_kind=oracle.PRED_V)
        np.testing.assert_allclose(math.sqrt(ab) * xt - math.sqrt(1 - ab) * v, x0, atol=1e-12)
        # the last step (alpha-bar 1) lands on x0
        xn1, _ = oracle.reconstruct(xt, x0, oracle.DDIM, a_t=ab, a_prev=1.0)
        np.testing.assert_allclose(xn1, x0, atol=1e-13)
        # a proper DDIM step re-noises x0 with the same eps
        xn2, _ = oracle.reconstruct(xt, x0, oracle.DDIM, a_t=ab, a_prev=0.99)
        np.testing.assert_allclose(xn2, math.sqrt(0.99) * x0 + math.sqrt(0.01) * eps0, atol=1e-11)


def test_flow_matching_euler_closed_form():
    rng = np.random.default_rng(2)
    x0 = rng.standard_normal(1000)
    eps0 = rng.standard_normal(1000)
    for s, s2 in ((1.0, 0.98), (0.5, 0.25), (0.02, 0.0)):
        xs = (1 - s) * x0 + s * eps0
        xn, vel = oracle.reconstruct(xs, x0, oracle.FM_EULER, sigma=s, sigma_next=s2,
                                     pred_kind=oracle.PRED_VELOCITY)
        np.testing.assert_allclose(vel, eps0 - x0, atol=1e-12 / s)
        # along the straight path the Euler step is exact
        np.testing.assert_allclose(xn, (1 - s2) * x0 + s2 * eps0, atol=1e-11)
    with pytest.raises(ValueError):
        oracle.reconstruct(x0, x0, oracle.FM_EULER, sigma=0.0, sigma_next=0.0)


def test_all_anchor_step_equals_stock_sampler(workloads):
    # a = N: every view is an anchor, the step must equal the stock sampler
    # step bit for bit (the paper's correctness gate, Sec. 3.2)
    w = workloads("hunyuan64")
    anchors = list(range(w.N))
    x0_prev, x0_new = _setup(w, anchors)
    xt = np.random.default_rng(5).standard_normal(x0_prev.shape)
    r = dict(sampler=oracle.DDIM, a_t=0.3, a_prev=0.4)
    x0_out, xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, x_t=xt, recon=r,
                                          geom=(w.pos, w.valid, w.cams, oracle.tau(w.pos, w.valid)))
    np.testing.assert_array_equal(x0_out, x0_new)
    ref, _ = oracle.reconstruct(xt, x0_new, oracle.DDIM, a_t=0.3, a_prev=0.4)
    np.testing.assert_array_equal(xn, ref)


# ------------------------------------------------------------------ bf16 --
def test_bf16_rounding_definition():
    import torch
    rng = np.random.default_rng(4)
    x = np.concatenate([rng.standard_normal(10000) * s for s in (1e-3, 1.0, 1e3)]).astype(np.float32)
    x = np.concatenate([x, np.float32([0.0, -0.0, 1e-40, -3e-39, 3.3e38, 65504.0])])
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.round_bf16(x.astype(np.float64)), ref)
    # ties to even
    assert oracle.round_bf16([1 + 2 ** -8])[0] == 0x3F80
    assert oracle.round_bf16([1 + 3 * 2 ** -8])[0] == 0x3F82
    assert oracle.round_bf16([-(1 + 2 ** -8 + 2 ** -30)])[0] == 0xBF81
    assert oracle.round_bf16([1e39])[0] == 0x7F80
    assert oracle.round_bf16([float("nan")])[0] & 0x7FFF > 0x7F80


# --------------------------------------------------- rotation / schedule --
def test_rotation_tiny_and_coverage():
    # the tiny workload's first cached step has anchors {0, 3}
    assert oracle.rotate_anchors(6, 2, 0) == [0, 3]
    for N, a in ((6, 2), (6, 3), (12, 4), (10, 2), (6, 4), (6, 6), (7, 3)):
        s = -(-N // a)
        seen = set()
        for r in range(s):
            A = oracle.rotate_anchors(N, a, r)
            assert len(A) == a and len(set(A)) == a and all(0 <= x < N for x in A)
            assert A == sorted(A)
            seen |= set(A)
        # every view returns to the anchor set within ceil(N/a) cached steps
        assert seen == set(range(N)), (N, a)
        if N % a == 0:  # and exactly once
            cnt = np.zeros(N, int)
            for r in range(s):
                cnt[oracle.rotate_anchors(N, a, r)] += 1
            assert (cnt == 1).all()


def test_schedules():
    hmt = {"kind": "head_mid_tail", "head": 2, "mid": 1, "tail": 1}
    assert [t for t in range(10) if oracle.is_full_step(t, 10, hmt)] == [0, 1, 5, 9]
    ek = {"kind": "every_k", "k": 5}
    assert [t for t in range(30) if oracle.is_full_step(t, 30, ek)] == [0, 5, 10, 15, 20, 25]
    assert oracle.cached_ordinal(7, 30, ek) == 5
    assert [oracle.is_full_step(t, 1, {"kind": "single_cached"}) for t in range(2)] == [True, False]


def _table1():
    rows = []
    with open(os.path.join(GOLDEN, "table1_flops.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                b, st, ss, N, a, S, full, printed, name = line.split()
                rows.append((b, float(st), int(ss), int(N), int(a), int(S), int(full), float(printed), name))
    return rows


@pytest.mark.parametrize("row", _table1(), ids=lambda r: r[0] + "_" + r[-1])
def test_cost_model_reproduces_table1(row):
    # Table 1 FLOPs: a full step costs the stock per-step cost and a cached
    # step a/N of it; each printed figure solves to a whole number of full steps
    b, stock, ssteps, N, a, S, full, printed, _ = row
    per = stock / ssteps
    if b == "hunyuan" and full == 4:
        sched = {"kind": "head_mid_tail", "head": 2, "mid": 1, "tail": 1}  # the text's schedule
    else:
        sched = {"kind": "list", "steps": list(range(full - 1)) + [S - 1]}
    assert sum(oracle.is_full_step(t, S, sched) for t in range(S)) == full
    assert oracle.denoiser_flops(S, N, a, sched, per) == pytest.approx(printed, abs=0.006)


# --------------------------------------------------- anchor-row pack / unpack --
def test_pack_unpack_pins():
    rng = np.random.default_rng(9)
    x = rng.standard_normal((3, 6, 4, 5, 7))
    A = [1, 4]
    p = oracle.pack_anchors(x, A)
    assert p.shape == (3, 2, 4, 5, 7)
    for b in range(3):  # row by row, the definition
        for s, u in enumerate(A):
            np.testing.assert_array_equal(p[b, s], x[b, u])
    # all views as anchors: identity; unpack inverts pack on the anchor rows and
    # leaves the others untouched
    np.testing.assert_array_equal(oracle.pack_anchors(x, range(6)), x)
    y = rng.standard_normal(x.shape)
    z = oracle.unpack_anchors(p, y, A)
    np.testing.assert_array_equal(z[:, A], x[:, A])
    others = [v for v in range(6) if v not in A]
    np.testing.assert_array_equal(z[:, others], y[:, others])
