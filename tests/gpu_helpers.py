"""Shared plumbing of the GPU tests: seeded step inputs, device uploads and
the parity tolerances.

Tolerances (from the required bar: latents within 1e-5 relative in fp32 and
2e-2 absolute in bf16; indices bit-exact):
* fp32 values (x0 cache, fp32 latents, weights): |gpu - ref| <= 1e-5 * max(|ref|, 1).
  This is how the stated "1e-5 relative" is read: relative to |ref| where
  |ref| >= 1 and relative to unit scale below it.  The floor is needed
  because latents are unit-variance and a transported sum can cancel to ~0,
  where a purely relative bound is meaningless; the kernels' float
  arithmetic errs by a few ulp of the operands (<1e-6 at unit scale).  The
  largest purely relative error over |ref| >= 1e-2 is reported beside it.
* bf16 latents: |gpu - ref| <= 2e-2 against the oracle's unrounded binary64
  value, and, where |ref| >= 2^-6, at most one bf16 ulp away from the
  oracle's own rounding (the kernel rounds a float result, the oracle a
  binary64 one, so a tie can land one ulp apart; below 2^-6 a bf16 ulp is
  smaller than the float error of a sum of unit-scale terms, so only the
  absolute bound applies there).
* predictions (eps, v): the conversion divides by sqrt(1 - ab_t), which
  magnifies the error of x0 by sqrt(ab_t)/sqrt(1 - ab_t); the bound is
  1e-5 * (1 + sqrt(ab_t)/sqrt(1 - ab_t)) * max(|ref|, 1).
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2608_13255_gb300 import synth

RTOL = 1e-5
BF16_ATOL = 2e-2


REL_FLOOR = 1e-2  # |ref| above which the purely relative error is reported


def max_rel_err(got, ref, floor=REL_FLOOR):
    """Largest |got - ref| / |ref| over the elements with |ref| >= floor (0 if none)."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    big = np.abs(ref) >= floor
    if not big.any():
        return 0.0
    return float((np.abs(got - ref)[big] / np.abs(ref[big])).max())


def assert_f32_close(got, ref, scale=1.0, what=""):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(got - ref)
    bound = RTOL * scale * np.maximum(np.abs(ref), 1.0)
    bad = err > bound
    rel = max_rel_err(got, ref)
    assert not bad.any(), "%s: %d/%d outside tolerance, worst %.3g at %s (got %r, ref %r); max rel err %.3g" % (
        what, bad.sum(), bad.size, err.max(), np.unravel_index(err.argmax(), err.shape),
        got.reshape(-1)[err.argmax()], ref.reshape(-1)[err.argmax()], rel)
    print("%s: max |err| %.3g, max rel err %.3g over |ref| >= %g" % (what or "f32", err.max(), rel, REL_FLOOR))
    return float(err.max())


def bf16_to_f64(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _ordered(bits):
    b = np.asarray(bits, np.uint16).astype(np.int32)
    return np.where(b & 0x8000, 0x8000 - b, b)  # monotone integer order of bf16 values


def assert_bf16_close(got_bits, ref64, what=""):
    got = bf16_to_f64(got_bits)
    err = np.abs(got - ref64)
    assert err.max() <= BF16_ATOL, "%s: max |err| %.4g > %.3g" % (what, err.max(), BF16_ATOL)
    ulps = np.abs(_ordered(got_bits) - _ordered(oracle.round_bf16(ref64)))
    ulps = np.where(np.abs(ref64) >= 2.0 ** -6, ulps, 0)
    bad = ulps > 1
    assert not bad.any(), "%s: %d elements more than one bf16 ulp from the oracle (e.g. got %r ref %r)" % (
        what, bad.sum(), got[bad][:3], ref64[bad][:3])
    return float(err.max()), float((ulps == 1).mean())


def lat_torch_dtype(w):
    return torch.bfloat16 if w.dtype == "bf16" else torch.float32


def latent_values(x32, w):
    """Latent array as the GPU stores it (bf16-rounded for bf16 workloads),
    returned as float64 values for the oracle and as a torch tensor."""
    if w.dtype == "bf16":
        bits = synth.to_bf16_bits(x32)
        t = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16)
        return bf16_to_f64(bits), t
    return x32.astype(np.float64), torch.from_numpy(np.ascontiguousarray(x32))


def step_inputs(w, step, anchors, seed_extra=0):
    """x0_prev [B,N,C,H,W] f32, x0_new [B,a,C,H,W] f32 and x_t (float32 before
    storage rounding) for one step of a workload."""
    rng = np.random.default_rng(np.random.SeedSequence([w.seed, 77, step, seed_extra]))
    shp = (w.B, w.N, w.C, w.H, w.W)
    x0_prev = rng.standard_normal(shp, dtype=np.float32)
    x0_new = x0_prev[:, anchors] + synth.delta(w, step, anchors)
    x_t = rng.standard_normal(shp, dtype=np.float32)
    return x0_prev, np.ascontiguousarray(x0_new, dtype=np.float32), x_t


def recon_kw(params, pred=None):
    """Arguments for the oracle's reconstruction from a synth.recon_params dict."""
    r = dict(sampler=oracle.DDIM if params["sampler"] == "ddim" else oracle.FM_EULER,
             a_t=params.get("a_t", 0.0), a_prev=params.get("a_prev", 0.0),
             sigma=params.get("sigma", 0.0), sigma_next=params.get("sigma_next", 0.0),
             pred_kind={None: 0, "eps": 1, "v": 2, "velocity": 3}[pred])
    return r


def pred_scale(params):
    if params["sampler"] == "ddim":
        a = params["a_t"]
        return 1.0 + math.sqrt(a) / math.sqrt(1.0 - a)
    return 1.0 + 1.0 / params["sigma"]


class DeviceGeometry:
    """A workload's geometry on the GPU, with tau, the keep masks and
    (optionally) the idx/w tables, built by geocache_build_corr.  `corr`
    uses the keep masks (the fast path); corr_for(mode) gives the others."""

    def __init__(self, w, K=4, tables=True, dev="cuda", source_index=True):
        from paper_2608_13255_gb300 import geocache as gc
        self.gc = gc
        self.w = w
        self.K = K
        self.pos = torch.from_numpy(w.pos).to(dev)
        self.valid = torch.from_numpy(w.valid).to(dev)
        self.cams = torch.from_numpy(w.cams).to(dev)
        self.tau = torch.zeros(w.B, dtype=torch.float32, device=dev)
        self.idx = self.wt = None
        if tables:
            shp = (w.B, w.N, w.N, w.H, w.W, K)
            self.idx = torch.empty(shp, dtype=torch.int32, device=dev)
            self.wt = torch.empty(shp, dtype=torch.float32, device=dev)
        self.keep = torch.empty((w.B, w.N, w.N, w.H, w.W), dtype=torch.uint8, device=dev)
        self.tile_ptr = torch.empty(w.B * w.N * w.N * gc.tiles_per_view(w.H, w.W) + 1, dtype=torch.int32,
                                    device=dev)
        c0 = gc.make_corr(self.pos, self.valid, self.cams, self.tau, K=K, tol_frac=w.tol_frac, keep=self.keep,
                          tile_ptr=self.tile_ptr, mode=gc.CORR_MASK)
        self.n_records = gc.record_count(c0)
        self.records = torch.empty((max(self.n_records, 1), 4), dtype=torch.int32, device=dev)
        # source index of the records (used by sparse steps with C >= 8)
        self.src_ptr = self.src_rec = None
        if source_index:
            self.src_ptr = torch.empty(w.B * w.N * gc.tiles_per_view(w.H, w.W) + 1, dtype=torch.int32, device=dev)
            self.src_rec = torch.empty((self.records.shape[0], 2), dtype=torch.int32, device=dev)
        self.corr = gc.make_corr(self.pos, self.valid, self.cams, self.tau, self.idx, self.wt, K=K,
                                 tol_frac=w.tol_frac, keep=self.keep, tile_ptr=self.tile_ptr, records=self.records,
                                 mode=gc.CORR_SPARSE, src_ptr=self.src_ptr, src_rec=self.src_rec)
        gc.build_corr(self.corr)

    def corr_for(self, mode):
        """The corr in another mode; 'sparse_plain' is the sparse form without
        its source index (the record-parallel apply at any C)."""
        gc = self.gc
        m = {"mask": gc.CORR_MASK, "geometry": gc.CORR_GEOMETRY, "table": gc.CORR_TABLE,
             "sparse": gc.CORR_SPARSE, "sparse_plain": gc.CORR_SPARSE}[mode]
        src = mode == "sparse"
        return gc.make_corr(self.pos, self.valid, self.cams, self.tau, self.idx, self.wt, K=self.K,
                            tol_frac=self.w.tol_frac, keep=self.keep, tile_ptr=self.tile_ptr, records=self.records,
                            mode=m, src_ptr=self.src_ptr if src else None, src_rec=self.src_rec if src else None)

    def workspace(self, C, minimal=False):
        """Scratch for a sparse step: the fastest path's size, or (minimal)
        the smallest one a step accepts, max_records * C floats, which leaves
        no room for the increment plane of wide latents."""
        n = self.corr.min_workspace_floats(C) if minimal else self.corr.workspace_floats(C)
        return torch.empty(max(n, 4), dtype=torch.float32, device=self.pos.device)
