"""GeoCache CPU ORACLE -- test infrastructure, not product code.

Plain, slow, obviously-correct restatement of the paper's geometric delta
transport (Sec. 3.2), used only by ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py``.  The numeric core is the plain C file
``geocache_oracle.c`` (compiled with gcc, ``-ffp-contract=off``); the anchor
rotation, the refresh schedule and the trajectory loop are plain Python below.
Nothing here imports or links the CUDA path.

Pins (tests that tie this oracle to the paper and to mathematics rather than
to itself) live in ``tests/test_oracle_*.py``.  Every function below is
pinned; none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = None

DDIM, FM_EULER = 0, 1
PRED_NONE, PRED_EPS, PRED_V, PRED_VELOCITY = 0, 1, 2, 3

_P = ctypes.c_void_p


def build(force: bool = False) -> str:
    """Compile the oracle's C core (host gcc; no CUDA)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    src = os.path.join(_HERE, "geocache_oracle.c")
    out = os.path.join(_LIBDIR, "libgeocache_oracle.so")
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
                               "-shared", "-fPIC", "-o", tmp, src, "-lm"])
        os.replace(tmp, out)
    return out


def _lib():
    global _LIB
    if _LIB is None:
        lib = ctypes.CDLL(build())
        i, f, d, l = ctypes.c_int, ctypes.c_float, ctypes.c_double, ctypes.c_long
        lib.oracle_tau.argtypes = [_P, _P, i, i, i, i, f, _P]
        lib.oracle_tau.restype = i
        lib.oracle_project.argtypes = [_P, _P, _P, _P]
        lib.oracle_project.restype = i
        lib.oracle_taps.argtypes = [_P, _P, _P, i, i, _P, f, i, _P, _P, _P]
        lib.oracle_taps.restype = i
        lib.oracle_build_corr.argtypes = [_P, _P, _P, _P, i, i, i, i, i, _P, _P, _P]
        lib.oracle_build_corr.restype = l
        lib.oracle_brute_row.argtypes = [_P, _P, _P, i, i, _P, f, i, _P, _P]
        lib.oracle_brute_row.restype = i
        lib.oracle_reconstruct.argtypes = [_P, _P, _P, _P, l, i, d, d, d, d, i]
        lib.oracle_reconstruct.restype = i
        lib.oracle_transport_step.argtypes = [i, i, i, i, i, i, _P, _P, _P, _P, _P, _P, _P, i,
                                              _P, _P, _P, _P, _P, _P, i, d, d, d, d, i, _P, i]
        lib.oracle_transport_step.restype = i
        lib.oracle_raster.argtypes = [_P, i, _P, i, _P, i, i, _P, _P]
        lib.oracle_raster.restype = i
        lib.oracle_pool.argtypes = [_P, _P, i, i, i, _P, _P]
        lib.oracle_pool.restype = i
        lib.oracle_round_bf16.argtypes = [_P, _P, l]
        lib.oracle_round_bf16.restype = None
        _LIB = lib
    return _LIB


def _c(x, dtype):
    return np.ascontiguousarray(x, dtype=dtype)


def _ptr(x):
    return None if x is None else x.ctypes.data


# --------------------------------------------------------------- geometry --
def tau(pos, valid, tol_frac=0.01):
    """tau per asset: tol_frac x diagonal of the foreground texels' box."""
    pos, valid = _c(pos, np.float32), _c(valid, np.uint8)
    B, N, H, W = valid.shape
    out = np.zeros(B, np.float32)
    rc = _lib().oracle_tau(pos.ctypes.data, valid.ctypes.data, B, N, H, W, tol_frac, out.ctypes.data)
    assert rc == 0
    return out


def project(cam, X):
    """(uu, vv) of world point X in camera `cam` (binary32), or None."""
    cam, X = _c(cam, np.float32), _c(X, np.float32)
    uu, vv = ctypes.c_float(), ctypes.c_float()
    ok = _lib().oracle_project(cam.ctypes.data, X.ctypes.data, ctypes.byref(uu), ctypes.byref(vv))
    return (uu.value, vv.value) if ok else None


def build_corr(pos, valid, cams, tau_b, K=4, with_band=True):
    """Correspondence tables idx [B,N,N,H,W,K] i32, w f64, band [B,N,N,H,W] u8."""
    pos, valid, cams, tau_b = _c(pos, np.float32), _c(valid, np.uint8), _c(cams, np.float32), _c(tau_b, np.float32)
    B, N, H, W = valid.shape
    idx = np.empty((B, N, N, H, W, K), np.int32)
    w = np.empty((B, N, N, H, W, K), np.float64)
    band = np.zeros((B, N, N, H, W), np.uint8) if with_band else None
    n = _lib().oracle_build_corr(pos.ctypes.data, valid.ctypes.data, cams.ctypes.data, tau_b.ctypes.data,
                                 B, N, H, W, K, idx.ctypes.data, w.ctypes.data, _ptr(band))
    assert n >= 0
    return idx, w, band


def brute_row(cam_u, pos_u, valid_u, X, tau_v, K=4):
    """Brute-force row of G_{u->v} for target point X: list of (q, w)."""
    cam_u, pos_u, valid_u, X = (_c(cam_u, np.float32), _c(pos_u, np.float32),
                                _c(valid_u, np.uint8), _c(X, np.float32))
    H, W = valid_u.shape
    q = np.zeros(4, np.int32)
    w = np.zeros(4, np.float64)
    n = _lib().oracle_brute_row(cam_u.ctypes.data, pos_u.ctypes.data, valid_u.ctypes.data, H, W,
                                X.ctypes.data, float(tau_v), K, q.ctypes.data, w.ctypes.data)
    assert n >= 0
    return list(zip(q[:n].tolist(), w[:n].tolist()))


def taps(cam_u, pos_u, valid_u, X, tau_v, K=4):
    """Tap table row (idx[K], w[K]) for target point X in source view u."""
    cam_u, pos_u, valid_u, X = (_c(cam_u, np.float32), _c(pos_u, np.float32),
                                _c(valid_u, np.uint8), _c(X, np.float32))
    H, W = valid_u.shape
    idx = np.zeros(K, np.int32)
    w = np.zeros(K, np.float64)
    _lib().oracle_taps(cam_u.ctypes.data, pos_u.ctypes.data, valid_u.ctypes.data, H, W,
                       X.ctypes.data, float(tau_v), K, idx.ctypes.data, w.ctypes.data, None)
    return idx, w


# ---------------------------------------------------------- reconstruction --
def reconstruct(x_t, x0, sampler, a_t=0.0, a_prev=0.0, sigma=0.0, sigma_next=0.0, pred_kind=PRED_NONE):
    """Elementwise x_t, x0 -> (x_next, pred) in binary64."""
    x_t, x0 = _c(x_t, np.float64), _c(x0, np.float64)
    x_next = np.empty_like(x_t)
    pred = np.empty_like(x_t) if pred_kind else None
    rc = _lib().oracle_reconstruct(x_t.ctypes.data, x0.ctypes.data, x_next.ctypes.data, _ptr(pred),
                                   x_t.size, sampler, a_t, a_prev, sigma, sigma_next, pred_kind)
    if rc != 0:
        raise ValueError("invalid reconstruction parameters")
    return x_next, pred


# ------------------------------------------------------------- transport --
def transport_step(anchors, x0_new, x0_prev, *, K=4, table=None, geom=None,
                   x_t=None, recon=None, sel=None, update="delta"):
    """One cached step (Eq. 1 + aggregation + loop order of Sec. 3.2).

    table = (idx, w) tables, or geom = (pos, valid, cams, tau).
    recon = dict(sampler=..., a_t=, a_prev=, sigma=, sigma_next=, pred_kind=) or None.
    update = "delta" (Eq. 1) or "copy" (the value-copy ablation of Sec. 4.3:
    covered targets take the anchors' transported x0).
    Returns (x0_out, x_next, pred) in binary64 (x_next/pred None without recon).
    """
    if update not in ("delta", "copy"):
        raise ValueError("update must be 'delta' or 'copy'")
    x0_new, x0_prev = _c(x0_new, np.float64), _c(x0_prev, np.float64)
    B, N, C, H, W = x0_prev.shape
    a = len(anchors)
    anc = _c(sorted(anchors), np.int32).astype(np.intc)
    x0_out = np.zeros_like(x0_prev)
    x_next = pred = None
    r = dict(sampler=DDIM, a_t=0.0, a_prev=0.0, sigma=0.0, sigma_next=0.0, pred_kind=PRED_NONE)
    if recon is not None:
        r.update(recon)
        x_t = _c(x_t, np.float64)
        x_next = np.zeros_like(x0_prev)
        if r["pred_kind"]:
            pred = np.zeros_like(x0_prev)
    idx = w = pos = valid = cams = tau_b = None
    if table is not None:
        idx, w = _c(table[0], np.int32), _c(table[1], np.float64)
        K = idx.shape[-1]
    else:
        pos, valid, cams, tau_b = (_c(geom[0], np.float32), _c(geom[1], np.uint8),
                                   _c(geom[2], np.float32), _c(geom[3], np.float32))
    if sel is not None:
        sel = _c(sel, np.uint8)
    rc = _lib().oracle_transport_step(
        B, N, H, W, K, C, _ptr(idx), _ptr(w), _ptr(pos), _ptr(valid), _ptr(cams), _ptr(tau_b),
        anc.ctypes.data, a, x0_new.ctypes.data, x0_prev.ctypes.data, x0_out.ctypes.data,
        _ptr(x_t if recon is not None else None), _ptr(x_next), _ptr(pred),
        r["sampler"], r["a_t"], r["a_prev"], r["sigma"], r["sigma_next"], r["pred_kind"], _ptr(sel),
        1 if update == "copy" else 0)
    if rc != 0:
        raise ValueError("oracle_transport_step: invalid arguments (%d)" % rc)
    return x0_out, x_next, pred


def shuffle_rows(idx, w, perm):
    """The shuffled-correspondence ablation of Sec. 4.3 ("corr -> shuffled")
    on dense tables: the nonzero rows of every G_{u->v} (target tokens of view
    v with a kept tap in view u), enumerated in (b, v, u, token) order, are
    permuted: row number r takes the taps and weights of row number perm[r].
    perm must map the rows of each (b, v, u) onto themselves.  Returns new
    (idx, w); zero rows stay zero."""
    idx, w = np.asarray(idx), np.asarray(w)
    K = idx.shape[-1]
    flat_i, flat_w = idx.reshape(-1, K), w.reshape(-1, K)
    rows = np.flatnonzero((flat_i >= 0).any(axis=1))  # (b, v, u, token) order
    perm = np.asarray(perm, dtype=np.int64)
    if perm.shape != rows.shape:
        raise ValueError("perm has %d entries for %d nonzero rows" % (perm.size, rows.size))
    out_i, out_w = flat_i.copy(), flat_w.copy()
    out_i[rows] = flat_i[rows[perm]]
    out_w[rows] = flat_w[rows[perm]]
    return out_i.reshape(idx.shape), out_w.reshape(w.shape)


def raster(V, F, cam, H, W):
    """Position map [H,W,3] f32 and validity [H,W] u8 of mesh (V [nv,3]
    world, F [nf,3] vertex indices) seen by camera `cam` (16 floats): the
    nearest face whose projection contains the pixel centre, ties to the
    lower face index; decisions and position in binary32 (Sec. 3.1 position
    maps; see oracle_raster)."""
    V = _c(V, np.float32)
    F = _c(F, np.int32)
    cam = _c(cam, np.float32)
    pos = np.zeros((H, W, 3), np.float32)
    valid = np.zeros((H, W), np.uint8)
    rc = _lib().oracle_raster(V.ctypes.data, V.shape[0], F.ctypes.data, F.shape[0], cam.ctypes.data, H, W,
                              pos.ctypes.data, valid.ctypes.data)
    if rc != 0:
        raise ValueError("oracle_raster: %d" % rc)
    return pos, valid


def raster_views(V, F, cams, H, W):
    """raster() for each camera of cams [N,16]: ([N,H,W,3], [N,H,W])."""
    out = [raster(V, F, c, H, W) for c in np.asarray(cams).reshape(-1, 16)]
    return np.stack([o[0] for o in out]), np.stack([o[1] for o in out])


def pool(pos_hi, valid_hi, s):
    """Token-grid position map and validity from maps rendered at s times
    the token resolution: pos_hi [..., H*s, W*s, 3], valid_hi [..., H*s, W*s]
    -> ([..., H, W, 3] f32, [..., H, W] u8).  A token's position is the
    binary32 mean of its valid pixels' positions (row-major order); it is
    foreground when at least half of its s*s pixels are (see oracle_pool)."""
    pos_hi = _c(pos_hi, np.float32)
    valid_hi = _c(valid_hi, np.uint8)
    Hs, Ws = valid_hi.shape[-2:]
    if Hs % s or Ws % s or pos_hi.shape != valid_hi.shape + (3,):
        raise ValueError("maps of %s are not an s=%d super-sampling" % (valid_hi.shape, s))
    H, W = Hs // s, Ws // s
    lead = valid_hi.shape[:-2]
    pos = np.zeros(lead + (H, W, 3), np.float32)
    valid = np.zeros(lead + (H, W), np.uint8)
    ph, vh = pos_hi.reshape(-1, Hs, Ws, 3), valid_hi.reshape(-1, Hs, Ws)
    po, vo = pos.reshape(-1, H, W, 3), valid.reshape(-1, H, W)
    for k in range(ph.shape[0]):
        rc = _lib().oracle_pool(ph[k].ctypes.data, vh[k].ctypes.data, H, W, int(s), po[k].ctypes.data,
                                vo[k].ctypes.data)
        if rc != 0:
            raise ValueError("oracle_pool: %d" % rc)
    return pos, valid


def scaled_camera(cam, s):
    """The camera of an s-times finer pixel grid: focal lengths and principal
    point multiplied by s in binary32 (token (i, j) of the coarse grid covers
    pixels (i s .. i s + s - 1, j s .. j s + s - 1) of the fine one)."""
    c = np.array(cam, np.float32).reshape(-1, 16).copy()
    c[:, 12:16] = c[:, 12:16] * np.float32(s)
    return c.reshape(np.shape(cam))


def raster_supersampled(V, F, cams, H, W, s):
    """Token-grid maps of a mesh from renders at s times the token
    resolution: raster() with scaled_camera(cam, s) at (H s, W s), then
    pool().  cams [N,16] -> ([N,H,W,3], [N,H,W])."""
    hi = raster_views(V, F, scaled_camera(np.asarray(cams).reshape(-1, 16), s), H * s, W * s)
    return pool(hi[0], hi[1], s)


def round_bf16(x) -> np.ndarray:
    """binary64 -> bfloat16 bit patterns (uint16), round to nearest even."""
    x = _c(x, np.float64)
    out = np.empty(x.shape, np.uint16)
    _lib().oracle_round_bf16(x.ctypes.data, out.ctypes.data, x.size)
    return out


# ------------------------------------------------- rotation and schedule --
def rotate_anchors(N: int, a: int, ordinal: int, contiguous: bool = False):
    """Anchor set of the `ordinal`-th cached step (Sec. 3.2, batch-sliced
    anchor forward: the anchors rotate every step and each view returns to
    full context every ceil(N/a) steps).

    Strided reading: s = ceil(N/a), r = ordinal mod s,
    A = {(r + j s) mod N : j < a}; a repeated id is replaced by the smallest
    unused id.  Contiguous reading: A = {(ordinal*a + j) mod N : j < a}.
    """
    if not (1 <= a <= N):
        raise ValueError("need 1 <= a <= N")
    if contiguous:
        cand = [(ordinal * a + j) % N for j in range(a)]
    else:
        s = -(-N // a)
        r = ordinal % s
        cand = [(r + j * s) % N for j in range(a)]
    out = []
    for c in cand:
        if c in out:
            c = next(x for x in range(N) if x not in out and x not in cand)
        out.append(c)
    return sorted(out)


def is_full_step(step: int, S: int, sched: dict) -> bool:
    """Full (all-view) or cached step (drift-bounding schedule, Sec. 3.2).

    Step 0 is always full: no x0(t-1) exists yet.
      every_k:        full iff step % k == 0
      head_mid_tail:  the first `head` steps, step floor(S/2) if mid, the
                      last `tail` steps
      list:           full iff step in `steps`
      all_full:       every step (the a = N correctness gate)
      single_cached:  step 0 is the supplied initial state; step 1 is cached
    """
    kind = sched["kind"]
    if kind == "single_cached":
        return step == 0
    if step == 0:
        return True
    if kind == "every_k":
        return step % sched["k"] == 0
    if kind == "head_mid_tail":
        if step < sched.get("head", 2):
            return True
        if sched.get("mid", 1) and step == S // 2:
            return True
        return step >= S - sched.get("tail", 1)
    if kind == "list":
        return step in set(sched["steps"])
    if kind == "all_full":
        return True
    raise ValueError(kind)


def cached_ordinal(step: int, S: int, sched: dict) -> int:
    """Number of cached steps strictly before `step`."""
    return sum(0 if is_full_step(t, S, sched) else 1 for t in range(step))


def denoiser_flops(S: int, N: int, a: int, sched: dict, per_step: float) -> float:
    """Denoiser cost of a schedule: a full step costs per_step, a cached step
    a/N of it (only the anchor rows run the denoiser)."""
    return sum(per_step if is_full_step(t, S, sched) else per_step * a / N for t in range(S))


# ------------------------------------------------- anchor-row pack / unpack --
def pack_anchors(src, anchors):
    """Rows of the anchor views, in anchor order (Sec. 3.2, batch-sliced
    anchor forward: the denoiser runs on the anchor rows only, each keeping
    its structural indices).  src [B, N, ...] -> [B, a, ...]."""
    src = np.asarray(src)
    return src[:, list(anchors)].copy()


def unpack_anchors(src, dst, anchors):
    """Scatter of anchor rows back to their views: dst[:, anchors[s]] = src[:, s]."""
    out = np.array(dst, copy=True)
    out[:, list(anchors)] = np.asarray(src)
    return out
