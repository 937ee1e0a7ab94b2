"""Pins of the oracle's two ablation modes (Sec. 4.3, Table 3): the value copy
("delta -> copy") and the shuffled correspondence ("corr -> shuffled").

Value copy: a covered target takes the mean over its covering anchors of the
transported anchor x0; an uncovered one keeps its state.  Shuffled
correspondence: the nonzero rows of each G_{u->v} exchange their taps by a
permutation within the pair.  Both are checked against dense operators
assembled from brute-force rows, and against closed forms.
"""
import numpy as np
import pytest

import oracle
from paper_2608_13255_gb300 import synth

from test_oracle_transport import _dense_operator, _setup


def _small():
    w = synth.make_workload("hunyuan64", H=16, W=16)
    return w, np.float32([0.12])  # about one token at 16x16: many covered targets


@pytest.mark.parametrize("K", [4, 1])
def test_value_copy_matches_dense_brute_force_operator(K):
    w, tau = _small()
    anchors = [1, 4]
    x0_prev, x0_new = _setup(w, anchors, seed=5)
    x0_out, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, K=K, geom=(w.pos, w.valid, w.cams, tau),
                                         update="copy")
    both = 0
    for v in range(w.N):
        if v in anchors:
            np.testing.assert_array_equal(x0_out[0, v], x0_new[0, anchors.index(v)])
            continue
        Gs = [_dense_operator(w, tau[0], u, v, K) for u in anchors]
        cover = sum((G.sum(1) > 0).astype(float) for G in Gs)
        both += int((cover == 2).sum())
        for c in range(w.C):
            val = sum(G @ x0_new[0, s, c].reshape(-1) for s, G in enumerate(Gs))
            ref = np.where(cover > 0, val / np.maximum(cover, 1), x0_prev[0, v, c].reshape(-1))
            np.testing.assert_allclose(x0_out[0, v, c].reshape(-1), ref, atol=2e-6 * 8, rtol=0)
    assert both > 0


def test_value_copy_closed_forms(workloads):
    w = workloads("hunyuan64")
    tau = oracle.tau(w.pos, w.valid)
    geom = (w.pos, w.valid, w.cams, tau)
    anchors = [0, 3]
    x0_prev, x0_new = _setup(w, anchors, seed=9)
    # a constant anchor field is reproduced exactly on every covered target
    # (rows are stochastic), uncovered targets keep their state bit for bit
    const = np.full_like(x0_new, 0.625)
    out_c, _, _ = oracle.transport_step(anchors, const, x0_prev, geom=geom, update="copy")
    out_d, _, _ = oracle.transport_step(anchors, x0_prev[:, anchors] + 1.0, x0_prev, geom=geom)
    covered = np.abs(out_d - x0_prev - 1.0) < 1e-9  # delta of exactly +1 marks the covered targets
    others = [v for v in range(w.N) if v not in anchors]
    cov = covered[:, others]
    assert cov.any() and (~cov).any()
    np.testing.assert_allclose(out_c[:, others][cov], 0.625, atol=1e-12, rtol=0)
    np.testing.assert_array_equal(out_c[:, others][~cov], x0_prev[:, others][~cov])
    # with a zero previous state the copy and the delta transport coincide
    zero = np.zeros_like(x0_prev)
    new0 = x0_new - x0_prev[:, anchors]
    a, _, _ = oracle.transport_step(anchors, new0, zero, geom=geom, update="copy")
    b, _, _ = oracle.transport_step(anchors, new0, zero, geom=geom)
    np.testing.assert_array_equal(a, b)


def _pair_counts(idx):
    B, N = idx.shape[:2]
    return (idx >= 0).any(-1).reshape(B, N, N, -1).sum(-1).reshape(-1)


def test_shuffle_rows_identity_transposition_and_multiset():
    w, tau = _small()
    idx, wt, _ = oracle.build_corr(w.pos, w.valid, w.cams, tau, K=4, with_band=False)
    counts = _pair_counts(idx)
    R = int(counts.sum())
    i0, w0 = oracle.shuffle_rows(idx, wt, np.arange(R))
    np.testing.assert_array_equal(i0, idx)
    np.testing.assert_array_equal(w0, wt)
    # a transposition of the first two rows of the first non-trivial pair
    start = int(np.argmax(counts >= 2))
    r0 = int(counts[:start].sum())
    perm = np.arange(R)
    perm[[r0, r0 + 1]] = perm[[r0 + 1, r0]]
    i1, w1 = oracle.shuffle_rows(idx, wt, perm)
    rows = np.flatnonzero((idx.reshape(-1, 4) >= 0).any(1))
    changed = np.flatnonzero((i1.reshape(-1, 4) != idx.reshape(-1, 4)).any(1))
    assert set(changed) <= {rows[r0], rows[r0 + 1]}
    np.testing.assert_array_equal(i1.reshape(-1, 4)[rows[r0]], idx.reshape(-1, 4)[rows[r0 + 1]])
    np.testing.assert_array_equal(w1.reshape(-1, 4)[rows[r0 + 1]], wt.reshape(-1, 4)[rows[r0]])
    # a seeded permutation within pairs keeps each pair's multiset of rows
    perm = synth.pair_permutation(counts, seed=3)
    i2, w2 = oracle.shuffle_rows(idx, wt, perm)
    B, N = idx.shape[:2]
    for pair in range(B * N * N):
        a = idx.reshape(B * N * N, -1, 4)[pair]
        b = i2.reshape(B * N * N, -1, 4)[pair]
        np.testing.assert_array_equal((a >= 0).any(1), (b >= 0).any(1))  # same covered tokens
        ka = np.sort(a[(a >= 0).any(1)].view([("", a.dtype)] * 4), axis=0)
        kb = np.sort(b[(b >= 0).any(1)].view([("", b.dtype)] * 4), axis=0)
        np.testing.assert_array_equal(ka, kb)
    assert (perm != np.arange(R)).mean() > 0.5


def test_shuffled_transport_matches_permuted_dense_operator():
    w, tau = _small()
    anchors = [1, 4]
    x0_prev, x0_new = _setup(w, anchors, seed=11)
    idx, wt, _ = oracle.build_corr(w.pos, w.valid, w.cams, tau, K=4, with_band=False)
    perm = synth.pair_permutation(_pair_counts(idx), seed=7)
    shuf = oracle.shuffle_rows(idx, wt, perm)
    x0_out, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, table=shuf)
    # the same permutation applied to the nonzero rows of brute-force operators
    N, HW = w.N, w.H * w.W
    counts = _pair_counts(idx).reshape(N, N)
    starts = np.concatenate([[0], np.cumsum(counts.reshape(-1))])[:-1].reshape(N, N)
    for v in range(N):
        if v in anchors:
            continue
        Gs = []
        for u in anchors:
            G = _dense_operator(w, tau[0], u, v, 4)
            rows = np.flatnonzero(G.sum(1) > 0)
            assert rows.size == counts[v, u]
            local = perm[starts[v, u]:starts[v, u] + rows.size] - starts[v, u]
            Gp = G.copy()
            Gp[rows] = G[rows[local]]
            Gs.append(Gp)
        cover = sum((G.sum(1) > 0).astype(float) for G in Gs)
        for c in range(w.C):
            inc = sum(G @ (x0_new[0, s, c].reshape(-1) - x0_prev[0, u, c].reshape(-1))
                      for s, (u, G) in enumerate(zip(anchors, Gs)))
            ref = x0_prev[0, v, c].reshape(-1) + np.where(cover > 0, inc / np.maximum(cover, 1), 0.0)
            np.testing.assert_allclose(x0_out[0, v, c].reshape(-1), ref, atol=2e-6 * 8, rtol=0)
    # and it differs from the unshuffled transport
    base, _, _ = oracle.transport_step(anchors, x0_new, x0_prev, table=(idx, wt))
    assert np.abs(base - x0_out).max() > 1e-3
