"""Seeded synthetic inputs for the geometric delta transport.

This module stands in for the paper's asset pool (eval200: 100 GSO + 100
Objaverse objects, Sec. 4.1), which is not available here, and for the
pretrained denoiser (its per-step x0 predictions are replaced by seeded
Gaussian updates).  It produces, for a workload:

* meshes and analytic solids normalised into the unit ball,
* look-at pinhole cameras (the multi-view layouts of the paper's substrates:
  six views on the batch axis, Sec. 3.1),
* per-view position maps and validity masks, rendered on the CPU
  (the maps a geometry-conditioned pipeline already has, Sec. 3.2),
* latents x_T ~ N(0, 1), an initial x0 ~ N(0, 1), and per-step x0 updates
  delta ~ N(0, 0.1^2).

It holds none of the method's arithmetic (no correspondence, transport or
reconstruction); both the CPU oracle and the CUDA path consume its arrays.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = None

CAM_FLOATS = 16  # R[9], t[3], fx, fy, cx, cy


# ---------------------------------------------------------------------------
# native rasteriser
# ---------------------------------------------------------------------------
def build_raster(force: bool = False) -> str:
    """Compile raster.c into an in-tree shared object (gcc, host only)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    src = os.path.join(_HERE, "raster.c")
    out = os.path.join(_LIBDIR, "libgeosynth.so")
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, src, "-lm"])
        os.replace(tmp, out)
    return out


def _lib():
    global _LIB
    if _LIB is None:
        lib = ctypes.CDLL(build_raster())
        lib.synth_raster_mesh.restype = ctypes.c_int
        lib.synth_raster_mesh.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]
        _LIB = lib
    return _LIB


# ---------------------------------------------------------------------------
# shapes
# ---------------------------------------------------------------------------
def icosphere(subdiv: int):
    """Unit icosphere with 10*4^s + 2 vertices (s=4: 2562, s=6: 40962)."""
    p = (1.0 + 5.0 ** 0.5) / 2.0
    V = np.array([[-1, p, 0], [1, p, 0], [-1, -p, 0], [1, -p, 0],
                  [0, -1, p], [0, 1, p], [0, -1, -p], [0, 1, -p],
                  [p, 0, -1], [p, 0, 1], [-p, 0, -1], [-p, 0, 1]], dtype=np.float64)
    F = np.array([[0, 11, 5], [0, 5, 1], [0, 1, 7], [0, 7, 10], [0, 10, 11],
                  [1, 5, 9], [5, 11, 4], [11, 10, 2], [10, 7, 6], [7, 1, 8],
                  [3, 9, 4], [3, 4, 2], [3, 2, 6], [3, 6, 8], [3, 8, 9],
                  [4, 9, 5], [2, 4, 11], [6, 2, 10], [8, 6, 7], [9, 8, 1]], dtype=np.int64)
    V /= np.linalg.norm(V, axis=1, keepdims=True)
    for _ in range(subdiv):
        e = np.concatenate([F[:, [0, 1]], F[:, [1, 2]], F[:, [2, 0]]], axis=0)
        e.sort(axis=1)
        uniq, inv = np.unique(e, axis=0, return_inverse=True)
        inv = inv.reshape(-1)
        mid = V[uniq[:, 0]] + V[uniq[:, 1]]
        mid /= np.linalg.norm(mid, axis=1, keepdims=True)
        base = V.shape[0]
        V = np.concatenate([V, mid], axis=0)
        m = F.shape[0]
        a, b, c = F[:, 0], F[:, 1], F[:, 2]
        ab, bc, ca = base + inv[:m], base + inv[m:2 * m], base + inv[2 * m:]
        F = np.concatenate([np.stack([a, ab, ca], 1), np.stack([b, bc, ab], 1),
                            np.stack([c, ca, bc], 1), np.stack([ab, bc, ca], 1)], axis=0)
    return V, F.astype(np.int32)


def _vertex_neighbour_mean(F, values, nv):
    s = np.zeros(nv)
    cnt = np.zeros(nv)
    for i, j in ((0, 1), (1, 2), (2, 0), (1, 0), (2, 1), (0, 2)):
        np.add.at(s, F[:, i], values[F[:, j]])
        np.add.at(cnt, F[:, i], 1.0)
    return s / np.maximum(cnt, 1.0)


def blob_mesh(subdiv: int, sigma: float, rng: np.random.Generator, smooth_iters: int = 4):
    """Icosphere with smooth radial noise of standard deviation `sigma`.

    Per-vertex N(0,1) radial offsets are smoothed by `smooth_iters` rounds of
    uniform Laplacian smoothing (n <- (n + mean_of_neighbours) / 2), then
    rescaled to zero mean and std `sigma`.
    """
    V, F = icosphere(subdiv)
    n = rng.standard_normal(V.shape[0])
    for _ in range(smooth_iters):
        n = 0.5 * n + 0.5 * _vertex_neighbour_mean(F, n, V.shape[0])
    n = (n - n.mean()) / max(n.std(), 1e-12) * sigma
    V = V * (1.0 + n)[:, None]
    V /= np.max(np.linalg.norm(V, axis=1))
    return V, F


def torus_mesh(R: float = 0.6, r: float = 0.25, nu: int = 96, nv: int = 48):
    """Torus around the z axis, normalised into the unit ball."""
    u = np.arange(nu) * (2 * math.pi / nu)
    v = np.arange(nv) * (2 * math.pi / nv)
    uu, vv = np.meshgrid(u, v, indexing="ij")
    X = (R + r * np.cos(vv)) * np.cos(uu)
    Y = (R + r * np.cos(vv)) * np.sin(uu)
    Z = r * np.sin(vv)
    V = np.stack([X, Y, Z], -1).reshape(-1, 3) / (R + r)
    idx = np.arange(nu * nv).reshape(nu, nv)
    i1 = np.roll(idx, -1, axis=0)
    j1 = np.roll(idx, -1, axis=1)
    ij1 = np.roll(i1, -1, axis=1)
    F = np.concatenate([np.stack([idx, i1, ij1], -1).reshape(-1, 3),
                        np.stack([idx, ij1, j1], -1).reshape(-1, 3)], 0)
    return V, F.astype(np.int32)


@dataclass
class Solids:
    """Union of analytic spheres and axis-aligned boxes (ray-cast exactly)."""
    spheres: list = field(default_factory=list)  # (centre[3], radius)
    boxes: list = field(default_factory=list)    # (centre[3], half[3])


def random_solids(rng: np.random.Generator, n_min: int = 3, n_max: int = 5) -> Solids:
    """3-5 boxes/spheres, centres U[-0.5,0.5]^3, half-sizes U[0.15,0.4],
    scaled so the union lies in the unit ball."""
    n = int(rng.integers(n_min, n_max + 1))
    s = Solids()
    reach = 0.0
    for _ in range(n):
        c = rng.uniform(-0.5, 0.5, 3)
        if rng.uniform() < 0.5:
            r = float(rng.uniform(0.15, 0.4))
            s.spheres.append((c, r))
            reach = max(reach, np.linalg.norm(c) + r)
        else:
            h = rng.uniform(0.15, 0.4, 3)
            s.boxes.append((c, h))
            reach = max(reach, np.linalg.norm(np.abs(c) + h))
    k = 1.0 / reach
    s.spheres = [(c * k, r * k) for c, r in s.spheres]
    s.boxes = [(c * k, h * k) for c, h in s.boxes]
    return s


def unit_sphere() -> Solids:
    return Solids(spheres=[(np.zeros(3), 1.0)])


# ---------------------------------------------------------------------------
# cameras
# ---------------------------------------------------------------------------
FOV_DEG = 40.0
CAM_DIST = 1.05 / math.sin(math.radians(FOV_DEG / 2))


def look_at_camera(az_deg: float, el_deg: float, H: int, W: int,
                   dist: float = CAM_DIST, fov_deg: float = FOV_DEG) -> np.ndarray:
    """Pinhole camera on a sphere of radius `dist`, looking at the origin.

    World +z is up; at the poles the up vector is (cos az, sin az, 0).
    Returns the 16-float record R[9], t[3], fx, fy, cx, cy (float32).
    """
    az, el = math.radians(az_deg), math.radians(el_deg)
    c = dist * np.array([math.cos(el) * math.cos(az), math.cos(el) * math.sin(az), math.sin(el)])
    f = -c / np.linalg.norm(c)
    up = np.array([0.0, 0.0, 1.0])
    if abs(abs(el_deg) - 90.0) < 1e-9:
        up = np.array([math.cos(az), math.sin(az), 0.0])
    right = np.cross(f, up)
    right /= np.linalg.norm(right)
    down = np.cross(f, right)
    Rm = np.stack([right, down, f], 0)
    t = -Rm @ c
    focal = (H / 2.0) / math.tan(math.radians(fov_deg / 2))
    rec = np.concatenate([Rm.reshape(-1), t, [focal, focal, W / 2.0, H / 2.0]])
    return rec.astype(np.float32)


def camera_aligned_plane(H: int, W: int, focal: float = 64.0, depth: float = 4.0, radius_frac: float = 0.4):
    """A fronto-parallel plane whose position map projects exactly onto the
    token centres: camera R = I, t = (0, 0, depth / 2), focal length `focal`
    (a power of two), principal point (W/2, H/2); token (i, j) holds the point
    of its centre ray at camera depth `depth`, ((i + 0.5 - W/2) depth / focal,
    (j + 0.5 - H/2) depth / focal, depth / 2).  Every coordinate and every step
    of its projection is exact in binary32, so the projection is exactly
    (i + 0.5, j + 0.5).  Foreground: tokens whose centre lies within
    radius_frac * min(H, W) of the image centre.
    Returns (cam [16] f32, pos [H, W, 3] f32, valid [H, W] u8)."""
    cam = np.zeros(CAM_FLOATS, np.float32)
    cam[[0, 4, 8]] = 1.0
    cam[11] = depth / 2.0
    cam[12:16] = (focal, focal, W / 2.0, H / 2.0)
    jj, ii = np.meshgrid(np.arange(H, dtype=np.float64), np.arange(W, dtype=np.float64), indexing="ij")
    du, dv = ii + 0.5 - W / 2.0, jj + 0.5 - H / 2.0
    pos = np.stack([du * depth / focal, dv * depth / focal, np.full_like(du, depth / 2.0)], -1).astype(np.float32)
    valid = (du * du + dv * dv <= (radius_frac * min(H, W)) ** 2).astype(np.uint8)
    pos[valid == 0] = 0.0
    return cam, pos, valid


def identity_camera_pair(w: "Workload", view: int = 0, plane: bool = False) -> "Workload":
    """A two-view workload whose views share one camera and one position map:
    view `view` of asset 0 of w (plane=False) or camera_aligned_plane (plane=True)."""
    if plane:
        cam, pos, valid = camera_aligned_plane(w.H, w.W)
    else:
        cam, pos, valid = w.cams[0, view], w.pos[0, view], w.valid[0, view]
    out = Workload(**{**w.__dict__})
    out.B, out.N, out.a = 1, 2, 1
    out.cams = np.ascontiguousarray(np.stack([cam, cam])[None], dtype=np.float32)
    out.pos = np.ascontiguousarray(np.stack([pos, pos])[None], dtype=np.float32)
    out.valid = np.ascontiguousarray(np.stack([valid, valid])[None], dtype=np.uint8)
    return out


def camera_centre(cam: np.ndarray) -> np.ndarray:
    R = cam[:9].astype(np.float64).reshape(3, 3)
    return -R.T @ cam[9:12].astype(np.float64)


def ring_layout(n: int, el_deg: float = 0.0):
    return [(360.0 * i / n, el_deg) for i in range(n)]


def hunyuan_layout():
    """Four azimuths at zero elevation plus top and bottom views."""
    return [(0.0, 0.0), (90.0, 0.0), (180.0, 0.0), (270.0, 0.0), (0.0, 90.0), (0.0, -90.0)]


def ring8_polar4_layout():
    """Ring of 8 alternating +-20 deg elevation plus 4 near-polar views."""
    ring = [(45.0 * i, 20.0 if i % 2 == 0 else -20.0) for i in range(8)]
    polar = [(0.0, 70.0), (180.0, 70.0), (90.0, -70.0), (270.0, -70.0)]
    return ring + polar


# ---------------------------------------------------------------------------
# rendering of position maps
# ---------------------------------------------------------------------------
def _pixel_rays(cam: np.ndarray, H: int, W: int):
    R = cam[:9].astype(np.float64).reshape(3, 3)
    fx, fy, cx, cy = (float(v) for v in cam[12:16])
    jj, ii = np.meshgrid(np.arange(H) + 0.5, np.arange(W) + 0.5, indexing="ij")
    d_cam = np.stack([(ii - cx) / fx, (jj - cy) / fy, np.ones_like(ii)], -1)  # [H,W,3]
    d_world = d_cam @ R  # R^T d for row vectors
    origin = camera_centre(cam)
    return origin, d_world


def cast_solids(solids: Solids, cam: np.ndarray, H: int, W: int):
    """Exact ray cast of the union of spheres and boxes through pixel centres."""
    o, d = _pixel_rays(cam, H, W)
    best = np.full((H, W), np.inf)
    for c, r in solids.spheres:
        oc = o - c
        b = d @ oc
        a = np.einsum("hwk,hwk->hw", d, d)
        cc = oc @ oc - r * r
        disc = b * b - a * cc
        ok = disc >= 0
        sq = np.sqrt(np.where(ok, disc, 0.0))
        t0 = (-b - sq) / a
        t1 = (-b + sq) / a
        t = np.where(t0 > 1e-9, t0, t1)
        t = np.where(ok & (t > 1e-9), t, np.inf)
        best = np.minimum(best, t)
    for c, h in solids.boxes:
        lo, hi = c - h, c + h
        with np.errstate(divide="ignore", invalid="ignore"):
            inv = 1.0 / d
            ta = (lo - o) * inv
            tb = (hi - o) * inv
        tmin = np.nanmax(np.minimum(ta, tb), axis=-1)
        tmax = np.nanmin(np.maximum(ta, tb), axis=-1)
        hit = (tmax >= tmin) & (tmax > 1e-9)
        t = np.where(tmin > 1e-9, tmin, tmax)
        best = np.minimum(best, np.where(hit, t, np.inf))
    valid = np.isfinite(best)
    P = o + d * np.where(valid, best, 0.0)[..., None]
    P = np.where(valid[..., None], P, 0.0)
    return P.astype(np.float32), valid.astype(np.uint8)


def raster_mesh(V: np.ndarray, F: np.ndarray, cam: np.ndarray, H: int, W: int):
    V = np.ascontiguousarray(V, dtype=np.float64)
    F = np.ascontiguousarray(F, dtype=np.int32)
    cam = np.ascontiguousarray(cam, dtype=np.float32)
    pos = np.zeros((H, W, 3), np.float32)
    valid = np.zeros((H, W), np.uint8)
    rc = _lib().synth_raster_mesh(V.ctypes.data, V.shape[0], F.ctypes.data, F.shape[0],
                                  cam.ctypes.data, H, W, pos.ctypes.data, valid.ctypes.data)
    if rc != 0:
        raise RuntimeError("synth_raster_mesh failed: %d" % rc)
    return pos, valid


def render_asset(shape, cams: np.ndarray, H: int, W: int):
    """Position maps [N,H,W,3] f32 and validity [N,H,W] u8 for one asset."""
    N = cams.shape[0]
    pos = np.zeros((N, H, W, 3), np.float32)
    valid = np.zeros((N, H, W), np.uint8)
    for v in range(N):
        if isinstance(shape, Solids):
            pos[v], valid[v] = cast_solids(shape, cams[v], H, W)
        else:
            pos[v], valid[v] = raster_mesh(shape[0], shape[1], cams[v], H, W)
    return pos, valid


# ---------------------------------------------------------------------------
# workloads
# ---------------------------------------------------------------------------
@dataclass
class Workload:
    name: str
    B: int
    N: int
    H: int
    W: int
    C: int
    a: int
    K: int
    dtype: str            # "f32" | "bf16" latent storage
    sampler: str          # "ddim" | "fm_euler"
    S: int                # sampler steps
    schedule: dict        # {"kind": "every_k", "k": 5} | {"kind": "head_mid_tail", ...} | {"kind": "single_cached"}
    layout: str
    mesh: str             # "sphere" | "blob2562" | "solids" | "blob40962" | "mixed"
    seed: int
    tol_frac: float = 0.01
    first_asset: int = 0        # global index of asset 0 (a shard of a larger batch starts there)
    cams: np.ndarray = None     # [B,N,16] f32
    pos: np.ndarray = None      # [B,N,H,W,3] f32
    valid: np.ndarray = None    # [B,N,H,W] u8

    @property
    def numel(self) -> int:
        return self.B * self.N * self.C * self.H * self.W


def _layout(name: str, N: int):
    if name == "ring6":
        return ring_layout(6)
    if name == "hunyuan6":
        return hunyuan_layout()
    if name == "ring8_polar4":
        return ring8_polar4_layout()
    raise ValueError(name)


def _shape_for(mesh: str, rng: np.random.Generator, asset: int):
    if mesh == "sphere":
        return unit_sphere()
    if mesh == "blob2562":
        return blob_mesh(4, 0.15, rng)
    if mesh == "blob40962":
        return blob_mesh(6, 0.15, rng)
    if mesh == "solids":
        return random_solids(rng)
    if mesh == "mixed":
        kind = asset % 3
        if kind == 0:
            return blob_mesh(4, 0.15, rng)
        if kind == 1:
            return random_solids(rng)
        return torus_mesh()
    raise ValueError(mesh)


WORKLOADS = {
    # unit sphere, 6-view ring, 32x32 fp32, anchors {0,3}, one DDIM step
    "tiny": dict(B=1, N=6, H=32, W=32, C=4, a=2, K=4, dtype="f32", sampler="ddim", S=1,
                 schedule={"kind": "single_cached"}, layout="ring6", mesh="sphere", seed=1001),
    # Hunyuan-style 6 views, blob (2562 verts), 64x64x4 bf16, 2 anchors, 30-step DDIM, full every 5
    "hunyuan64": dict(B=1, N=6, H=64, W=64, C=4, a=2, K=4, dtype="bf16", sampler="ddim", S=30,
                      schedule={"kind": "every_k", "k": 5}, layout="hunyuan6", mesh="blob2562", seed=1002),
    # 6 views, 96x96x4 bf16, boxes+spheres, 3 anchors, 50-step FM Euler, full every 4
    "solids96": dict(B=1, N=6, H=96, W=96, C=4, a=3, K=4, dtype="bf16", sampler="fm_euler", S=50,
                     schedule={"kind": "every_k", "k": 4}, layout="hunyuan6", mesh="solids", seed=1003),
    # 12 views (ring 8 +-20 deg + 4 polar), 128x128x16 bf16, blob 40962 verts, 4 anchors, 50-step Euler
    "ring12_128": dict(B=1, N=12, H=128, W=128, C=16, a=4, K=4, dtype="bf16", sampler="fm_euler", S=50,
                       schedule={"kind": "head_mid_tail", "head": 2, "mid": 1, "tail": 1},
                       layout="ring8_polar4", mesh="blob40962", seed=1004),
    # batch of independent assets x 6 views, 128x128x4 bf16 + f32 x0, mixed meshes, 2 anchors,
    # 30-step DDIM, full every 5 (B is swept; 8 is the base batch)
    "batch128": dict(B=8, N=6, H=128, W=128, C=4, a=2, K=4, dtype="bf16", sampler="ddim", S=30,
                     schedule={"kind": "every_k", "k": 5}, layout="hunyuan6", mesh="mixed", seed=1005),
}


def asset_seed(w_seed: int, asset: int, B: int) -> int:
    """Seed of the geometry of the asset with global index `asset` in a batch
    of B (a single-asset workload uses the workload seed itself)."""
    return w_seed if B == 1 else w_seed * 1000 + asset


def make_workload(name: str, **overrides) -> Workload:
    """Build a workload's geometry: cameras and rendered position maps."""
    spec = dict(WORKLOADS[name])
    spec.update(overrides)
    w = Workload(name=name, **spec)
    views = _layout(w.layout, w.N)
    assert len(views) == w.N, (name, len(views), w.N)
    cams1 = np.stack([look_at_camera(az, el, w.H, w.W) for az, el in views], 0)
    w.cams = np.ascontiguousarray(np.tile(cams1[None], (w.B, 1, 1)), dtype=np.float32)
    w.pos = np.zeros((w.B, w.N, w.H, w.W, 3), np.float32)
    w.valid = np.zeros((w.B, w.N, w.H, w.W), np.uint8)
    cache = {}
    single = w.B == 1 and w.first_asset == 0
    for b in range(w.B):
        g = w.first_asset + b  # global asset index
        s = asset_seed(w.seed, g, 1 if single else 2)
        # assets of the same mesh kind and seed render identically; cache by seed
        key = (w.mesh, s, g % 3 if w.mesh == "mixed" else 0)
        if key not in cache:
            rng = np.random.default_rng(s)
            shape = _shape_for(w.mesh, rng, g)
            cache[key] = render_asset(shape, w.cams[b], w.H, w.W)
        w.pos[b], w.valid[b] = cache[key]
    return w


def replicate_assets(w: Workload, B: int) -> Workload:
    """A workload with B assets cycling through w's rendered assets (for sweeps
    over batch size without re-rendering)."""
    idx = np.arange(B) % w.B
    out = Workload(**{**w.__dict__})
    out.B = B
    out.cams = np.ascontiguousarray(w.cams[idx])
    out.pos = np.ascontiguousarray(w.pos[idx])
    out.valid = np.ascontiguousarray(w.valid[idx])
    return out


# ---------------------------------------------------------------------------
# latents and the denoiser stand-in
# ---------------------------------------------------------------------------
def _rng(*key) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(k) for k in key]))


def initial_latents(w: Workload):
    """x_T ~ N(0,1) and x0 at step 0 ~ N(0,1), shape [B,N,C,H,W] float32.
    Each asset draws from its own stream, keyed by its global index, so a
    shard of a batch gets the same values as the whole batch."""
    shp = (w.N, w.C, w.H, w.W)
    xT = np.empty((w.B,) + shp, np.float32)
    x0 = np.empty((w.B,) + shp, np.float32)
    for b in range(w.B):
        g = w.first_asset + b
        xT[b] = _rng(w.seed, 0xA11CE, g).standard_normal(shp, dtype=np.float32)
        x0[b] = _rng(w.seed, 0x0B0B0, g).standard_normal(shp, dtype=np.float32)
    return xT, x0


def delta(w: Workload, step: int, views, std: float = 0.1) -> np.ndarray:
    """Per-step synthetic x0 update for the given views: [B,len(views),C,H,W]
    (one stream per step, view and global asset index)."""
    out = np.empty((w.B, len(views), w.C, w.H, w.W), np.float32)
    for b in range(w.B):
        g = w.first_asset + b
        for j, v in enumerate(views):
            out[b, j] = _rng(w.seed, 0xDE17A, step, v, g).standard_normal(
                (w.C, w.H, w.W), dtype=np.float32) * np.float32(std)
    return out


def pair_permutation(pair_counts, seed: int) -> np.ndarray:
    """Seeded input of the shuffled-correspondence ablation: a permutation of
    the records (int32) that maps the records of each (b, v, u) pair onto
    themselves; pair_counts[i] = records of pair i in (b, v, u) order."""
    counts = np.asarray(pair_counts, np.int64).reshape(-1)
    perm = np.empty(int(counts.sum()), np.int32)
    rng = _rng(0x5AFF1E, seed)
    start = 0
    for n in counts:
        perm[start:start + n] = start + rng.permutation(int(n))
        start += int(n)
    return perm


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round-to-nearest-even, via torch) and return
    the raw 16-bit patterns as uint16."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32)


# ---------------------------------------------------------------------------
# sampler noise schedules (properties of the substrate, inputs to the method)
# ---------------------------------------------------------------------------
def ddim_alpha_bars(S: int, T: int = 1000, beta_start: float = 0.00085, beta_end: float = 0.012):
    """alpha-bar at each of S DDIM steps and at the step after it.

    Scaled-linear betas over T training steps, timesteps round(linspace(T-1, 0, S)),
    and alpha-bar = 1 after the last step.  Returns float64 arrays (a_t, a_prev).
    """
    betas = np.linspace(beta_start ** 0.5, beta_end ** 0.5, T, dtype=np.float64) ** 2
    ab = np.cumprod(1.0 - betas)
    ts = np.round(np.linspace(T - 1, 0, S)).astype(np.int64)
    a_t = ab[ts]
    a_prev = np.append(ab[ts[1:]], 1.0)
    return a_t, a_prev


def fm_sigmas(S: int):
    """Linear flow-matching sigmas 1 -> 0: step k goes sigma_k -> sigma_{k+1}."""
    sig = 1.0 - np.arange(S + 1, dtype=np.float64) / S
    return sig[:-1], sig[1:]


def recon_params(w: "Workload", step: int) -> dict:
    """Sampler parameters of one step of a workload's trajectory."""
    if w.name == "tiny":
        return dict(sampler="ddim", a_t=0.5, a_prev=0.6)
    if w.sampler == "ddim":
        a_t, a_prev = ddim_alpha_bars(w.S)
        return dict(sampler="ddim", a_t=float(a_t[step]), a_prev=float(a_prev[step]))
    s, s_next = fm_sigmas(w.S)
    return dict(sampler="fm_euler", sigma=float(s[step]), sigma_next=float(s_next[step]))
