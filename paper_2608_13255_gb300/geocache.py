"""ctypes binding of libgeocache.so (include/geocache.h).

Same entry points as the C ABI; this module only marshals arguments (torch
tensors -> device pointers, dicts -> C structs, the current torch stream) and
checks that tensor shapes, dtypes and devices match what the C call will
read and write, since the C layer only sees pointers.  All computation runs
in the library's CUDA kernels; there is no fallback: if the library has not
been built, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

OK, EINVAL, ESHAPE, EDTYPE, ECUDA, ETIMEOUT, EDEVICE, EALIAS = 0, -1, -2, -3, -4, -5, -6, -7
F32, BF16 = 0, 1
DDIM, FM_EULER = 0, 1
PRED_NONE, PRED_EPS, PRED_V, PRED_VELOCITY = 0, 1, 2, 3
CORR_GEOMETRY, CORR_TABLE, CORR_MASK, CORR_SPARSE = 0, 1, 2, 3
UPDATE_DELTA, UPDATE_COPY = 0, 1
TILE_TOKENS = 1024
SCHED_EVERY_K, SCHED_HEAD_MID_TAIL, SCHED_LIST, SCHED_ALL_FULL, SCHED_SINGLE_CACHED = 0, 1, 2, 3, 4
MAX_VIEWS = 64

_SAMPLERS = {"ddim": DDIM, "fm_euler": FM_EULER, DDIM: DDIM, FM_EULER: FM_EULER}
_PREDS = {None: PRED_NONE, "none": PRED_NONE, "eps": PRED_EPS, "v": PRED_V, "velocity": PRED_VELOCITY,
          PRED_NONE: PRED_NONE, PRED_EPS: PRED_EPS, PRED_V: PRED_V, PRED_VELOCITY: PRED_VELOCITY}


class GeocacheError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__("geocache status %d: %s" % (status, msg))
        self.status = status


class Camera(ctypes.Structure):
    _fields_ = [("R", ctypes.c_float * 9), ("t", ctypes.c_float * 3), ("fx", ctypes.c_float),
                ("fy", ctypes.c_float), ("cx", ctypes.c_float), ("cy", ctypes.c_float)]


class Corr(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("N", ctypes.c_int), ("H", ctypes.c_int), ("W", ctypes.c_int),
                ("K", ctypes.c_int), ("tol_frac", ctypes.c_float),
                ("pos", ctypes.c_void_p), ("valid", ctypes.c_void_p), ("cams", ctypes.c_void_p),
                ("tau", ctypes.c_void_p), ("idx", ctypes.c_void_p), ("w", ctypes.c_void_p),
                ("keep", ctypes.c_void_p), ("tile_ptr", ctypes.c_void_p), ("records", ctypes.c_void_p),
                ("max_records", ctypes.c_int64), ("mode", ctypes.c_int),
                ("src_ptr", ctypes.c_void_p), ("src_rec", ctypes.c_void_p)]


class Recon(ctypes.Structure):
    _fields_ = [("sampler", ctypes.c_int), ("a_t", ctypes.c_double), ("a_prev", ctypes.c_double),
                ("sigma", ctypes.c_double), ("sigma_next", ctypes.c_double), ("pred_kind", ctypes.c_int),
                ("pred_out", ctypes.c_void_p)]


class Schedule(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("k", ctypes.c_int), ("head", ctypes.c_int), ("mid", ctypes.c_int),
                ("tail", ctypes.c_int), ("full_steps", ctypes.c_void_p), ("n_full_steps", ctypes.c_int),
                ("contiguous_rotation", ctypes.c_int)]


assert ctypes.sizeof(Camera) == 64

_LIB = None
EXPORTS = ("geocache_build_corr", "geocache_transport_step", "geocache_reconstruct", "geocache_is_full_step",
           "geocache_rotate_anchors", "geocache_device_status", "geocache_corr_record_count",
           "geocache_transport_workspace", "geocache_transport_step_noalloc", "geocache_pack_anchors",
           "geocache_unpack_anchors", "geocache_transport_step_update", "geocache_permute_records",
           "geocache_raster_posmaps", "geocache_debug_set_wait", "geocache_raster_posmaps_supersampled",
           "geocache_pool_posmaps",
           "geocache_last_error", "geocache_abi_version")


def lib_path() -> str:
    return _build.LIB


def load():
    """Load libgeocache.so; raise if it has not been built."""
    global _LIB
    if _LIB is None:
        path = lib_path()
        if not os.path.exists(path):
            raise RuntimeError("libgeocache.so is not built (%s); run __graft_entry__.build() or "
                               "python -m paper_2608_13255_gb300.build" % path)
        L = ctypes.CDLL(path)
        P, i, i64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64
        L.geocache_build_corr.argtypes = [ctypes.POINTER(Corr), P]
        L.geocache_transport_step.argtypes = [ctypes.POINTER(Corr), P, i, i, P, P, P, P, P, i,
                                              ctypes.POINTER(Recon), P, i64, P]
        L.geocache_transport_step_noalloc.argtypes = [ctypes.POINTER(Corr), P, i, i, P, P, P, P, P, i,
                                                      ctypes.POINTER(Recon), P]
        L.geocache_transport_step_noalloc.restype = ctypes.c_int
        L.geocache_transport_step_update.argtypes = [ctypes.POINTER(Corr), i, P, i, i, P, P, P, P, P, i,
                                                     ctypes.POINTER(Recon), P, i64, P]
        L.geocache_transport_step_update.restype = ctypes.c_int
        L.geocache_permute_records.argtypes = [ctypes.POINTER(Corr), P, P, P]
        L.geocache_permute_records.restype = ctypes.c_int
        L.geocache_raster_posmaps.argtypes = [P, i64, P, i64, P, i, P, i, i, i, P, P, P, P]
        L.geocache_raster_posmaps.restype = ctypes.c_int
        L.geocache_raster_posmaps_supersampled.argtypes = [P, i64, P, i64, P, i, P, i, i, i, i, P, P, P, P]
        L.geocache_raster_posmaps_supersampled.restype = ctypes.c_int
        L.geocache_pool_posmaps.argtypes = [P, P, i64, i, i, i, P, P, P]
        L.geocache_pool_posmaps.restype = ctypes.c_int
        for name in ("geocache_pack_anchors", "geocache_unpack_anchors"):
            getattr(L, name).argtypes = [P, P, i64, i, i, P, i, P]
            getattr(L, name).restype = ctypes.c_int
        L.geocache_corr_record_count.argtypes = [ctypes.POINTER(Corr), ctypes.POINTER(ctypes.c_int64), P]
        L.geocache_corr_record_count.restype = ctypes.c_int
        L.geocache_transport_workspace.argtypes = [ctypes.POINTER(Corr), i]
        L.geocache_transport_workspace.restype = ctypes.c_int64
        L.geocache_reconstruct.argtypes = [P, P, P, i, i64, ctypes.POINTER(Recon), P, P]
        L.geocache_is_full_step.argtypes = [i, i, ctypes.POINTER(Schedule)]
        L.geocache_rotate_anchors.argtypes = [i, i, i, i, ctypes.POINTER(Schedule), P, ctypes.POINTER(i)]
        L.geocache_device_status.argtypes = [P]
        L.geocache_debug_set_wait.argtypes = [ctypes.c_uint64, i]
        L.geocache_debug_set_wait.restype = ctypes.c_int
        L.geocache_last_error.restype = ctypes.c_char_p
        L.geocache_last_error.argtypes = []
        L.geocache_abi_version.argtypes = []
        for name in EXPORTS[:7]:
            getattr(L, name).restype = ctypes.c_int
        L.geocache_abi_version.restype = ctypes.c_int
        _LIB = L
    return _LIB


def last_error() -> str:
    return load().geocache_last_error().decode()


def _check(status: int):
    if status != OK:
        raise GeocacheError(status, last_error())
    return status


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _dev(t, dtype, numel=None, name="tensor"):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("%s must be a torch tensor" % name)
    if not t.is_cuda:
        raise ValueError("%s must be on a CUDA device" % name)
    if t.dtype != dtype:
        raise TypeError("%s must be %s (got %s)" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if numel is not None and t.numel() != numel:
        raise ValueError("%s has %d elements, expected %d" % (name, t.numel(), numel))
    return t.data_ptr()


def _lat_dtype(t):
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError("latents must be float32 or bfloat16 (got %s)" % t.dtype)


# ------------------------------------------------------------- structs --
class CorrHandle:
    """A filled geocache_corr plus references to the tensors it points to."""

    def __init__(self, c: Corr, keep):
        self.c = c
        self._keep = keep

    @property
    def tau(self):
        return self._keep["tau"]

    @property
    def idx(self):
        return self._keep.get("idx")

    @property
    def w(self):
        return self._keep.get("w")

    @property
    def keep(self):
        return self._keep.get("keep")

    def workspace_floats(self, C: int) -> int:
        """Workspace floats that select the fastest sparse path for C channels."""
        return load().geocache_transport_workspace(ctypes.byref(self.c), int(C))

    def min_workspace_floats(self, C: int) -> int:
        """The smallest workspace a sparse step with a < N accepts (max_records * C)."""
        return self.c.max_records * int(C) if self.c.mode == CORR_SPARSE else 0


def tiles_per_view(H: int, W: int) -> int:
    return -(-(H * W) // TILE_TOKENS)


def make_corr(pos, valid, cams, tau, idx=None, w=None, K=4, tol_frac=0.01, mode=None, keep=None,
              tile_ptr=None, records=None, src_ptr=None, src_rec=None) -> CorrHandle:
    """Describe a batch's geometry (and optional tables, keep masks and sparse
    form) for the C ABI.  records is an int32 tensor [R, 4] (16-byte tap
    records); src_ptr [B*N*T + 1] and src_rec [R, 2] int32 hold the optional
    source index.  The default mode is SPARSE when records are given, else MASK
    when keep masks are given, else TABLE when tables are given, else GEOMETRY."""
    B, N, H, W = valid.shape
    n = B * N * H * W
    refs = {"pos": pos, "valid": valid, "cams": cams, "tau": tau, "idx": idx, "w": w, "keep": keep,
            "tile_ptr": tile_ptr, "records": records, "src_ptr": src_ptr, "src_rec": src_rec}
    if mode is None:
        mode = (CORR_SPARSE if records is not None else CORR_MASK if keep is not None
                else CORR_TABLE if idx is not None else CORR_GEOMETRY)
    if records is not None and (records.dim() != 2 or records.shape[1] != 4):
        raise ValueError("records must be an int32 tensor of shape [R, 4]")
    c = Corr(B, N, H, W, K, tol_frac,
             _dev(pos, torch.float32, 3 * n, "pos"), _dev(valid, torch.uint8, n, "valid"),
             _dev(cams, torch.float32, 16 * B * N, "cams"), _dev(tau, torch.float32, B, "tau"),
             _dev(idx, torch.int32, n * N * K, "idx"), _dev(w, torch.float32, n * N * K, "w"),
             _dev(keep, torch.uint8, n * N, "keep"),
             _dev(tile_ptr, torch.int32, B * N * N * tiles_per_view(H, W) + 1, "tile_ptr"),
             _dev(records, torch.int32, None, "records"), 0 if records is None else records.shape[0], mode,
             _dev(src_ptr, torch.int32, B * N * tiles_per_view(H, W) + 1, "src_ptr"),
             _dev(src_rec, torch.int32, None if records is None else 2 * records.shape[0], "src_rec"))
    return CorrHandle(c, refs)


def record_count(corr: CorrHandle, stream=None) -> int:
    """geocache_corr_record_count (synchronous)."""
    n = ctypes.c_int64(0)
    _check(load().geocache_corr_record_count(ctypes.byref(corr.c), ctypes.byref(n), _stream(stream)))
    return int(n.value)


def build_sparse_corr(pos, valid, cams, K=4, tol_frac=0.01, tables=False, stream=None,
                      source_index=False) -> CorrHandle:
    """Allocate and build the full correspondence state of a batch: tau, keep
    masks, the sparse form (count, then records), optionally the tables and
    the source index (used by steps with 8 or more channels whose workspace
    has no room for the anchors' increment plane: they then apply the records
    per source tile).  Allocation happens here, once per batch of assets,
    never per step."""
    B, N, H, W = valid.shape
    dev = pos.device
    tau = torch.zeros(B, dtype=torch.float32, device=dev)
    keep = torch.empty((B, N, N, H, W), dtype=torch.uint8, device=dev)
    tile_ptr = torch.empty(B * N * N * tiles_per_view(H, W) + 1, dtype=torch.int32, device=dev)
    c0 = make_corr(pos, valid, cams, tau, K=K, tol_frac=tol_frac, keep=keep, tile_ptr=tile_ptr,
                   mode=CORR_MASK)
    R = record_count(c0, stream)
    records = torch.empty((max(R, 1), 4), dtype=torch.int32, device=dev)
    idx = w = None
    if tables:
        idx = torch.empty((B, N, N, H, W, K), dtype=torch.int32, device=dev)
        w = torch.empty((B, N, N, H, W, K), dtype=torch.float32, device=dev)
    src_ptr = src_rec = None
    if source_index:
        src_ptr = torch.empty(B * N * tiles_per_view(H, W) + 1, dtype=torch.int32, device=dev)
        src_rec = torch.empty((records.shape[0], 2), dtype=torch.int32, device=dev)
    corr = make_corr(pos, valid, cams, tau, idx=idx, w=w, K=K, tol_frac=tol_frac, keep=keep, tile_ptr=tile_ptr,
                     records=records, mode=CORR_SPARSE, src_ptr=src_ptr, src_rec=src_rec)
    return build_corr(corr, stream)


def make_recon(sampler="ddim", a_t=0.0, a_prev=0.0, sigma=0.0, sigma_next=0.0, pred_kind=None,
               pred_out=None) -> Recon:
    r = Recon(_SAMPLERS[sampler], float(a_t), float(a_prev), float(sigma), float(sigma_next),
              _PREDS[pred_kind], None if pred_out is None else _dev(pred_out, torch.float32, name="pred_out"))
    r._pred = pred_out  # keeps the tensor alive; its size is checked at the call
    return r


def _check_pred(recon, n):
    t = getattr(recon, "_pred", None) if recon is not None else None
    if t is not None and t.numel() != n:
        raise ValueError("pred_out has %d elements, expected %d" % (t.numel(), n))


_SCHED_KINDS = {"every_k": SCHED_EVERY_K, "head_mid_tail": SCHED_HEAD_MID_TAIL, "list": SCHED_LIST,
                "all_full": SCHED_ALL_FULL, "single_cached": SCHED_SINGLE_CACHED}


def make_schedule(spec: dict):
    kind = _SCHED_KINDS[spec["kind"]]
    steps = (ctypes.c_int32 * max(1, len(spec.get("steps", ()))))(*spec.get("steps", ()))
    s = Schedule(kind, int(spec.get("k", 1)), int(spec.get("head", 2)), int(spec.get("mid", 1)),
                 int(spec.get("tail", 1)), ctypes.cast(steps, ctypes.c_void_p), len(spec.get("steps", ())),
                 int(spec.get("contiguous", 0)))
    return s, steps


# ---------------------------------------------------------- entry points --
def build_corr(corr: CorrHandle, stream=None) -> CorrHandle:
    """geocache_build_corr: tau (and the tables if the handle has idx/w)."""
    _check(load().geocache_build_corr(ctypes.byref(corr.c), _stream(stream)))
    return corr


UPDATES = {"delta": UPDATE_DELTA, "copy": UPDATE_COPY}


def transport_step(corr: CorrHandle, anchors, C, x0_anchor_new, x0_prev, x0_out, x_t=None, x_next=None,
                   recon: Recon | None = None, workspace=None, stream=None, update="delta"):
    """geocache_transport_step (update="delta", Eq. 1) or
    geocache_transport_step_update (update="copy", the value-copy ablation)
    on torch tensors (see include/geocache.h)."""
    c = corr.c
    anc = sorted(int(a) for a in anchors)
    a = len(anc)
    n_all = c.B * c.N * C * c.H * c.W
    arr = (ctypes.c_int32 * max(1, a))(*anc)
    lat = F32
    pt = pn = None
    if recon is not None:
        lat = _lat_dtype(x_t)
        dt = x_t.dtype
        pt, pn = _dev(x_t, dt, n_all, "x_t"), _dev(x_next, dt, n_all, "x_next")
        _check_pred(recon, n_all)
    st = load().geocache_transport_step_update(
        ctypes.byref(c), UPDATES[update], ctypes.cast(arr, ctypes.c_void_p), a, int(C),
        _dev(x0_anchor_new, torch.float32, c.B * a * C * c.H * c.W, "x0_anchor_new"),
        _dev(x0_prev, torch.float32, n_all, "x0_prev"), _dev(x0_out, torch.float32, n_all, "x0_out"),
        pt, pn, lat, ctypes.byref(recon) if recon is not None else None,
        _dev(workspace, torch.float32, None, "workspace"), 0 if workspace is None else workspace.numel(),
        _stream(stream))
    _check(st)


def permute_records(corr: CorrHandle, perm, out=None, stream=None) -> CorrHandle:
    """geocache_permute_records (shuffled-correspondence ablation): a new
    sparse-mode handle over `out` (allocated like corr's records when None)
    whose rows exchange their taps by `perm` (device int32 [max_records])."""
    c = corr.c
    recs = corr._keep["records"]
    if out is None:
        out = torch.empty_like(recs)
    _check(load().geocache_permute_records(ctypes.byref(c), _dev(perm, torch.int32, c.max_records, "perm"),
                                           _dev(out, torch.int32, 4 * c.max_records, "out"), _stream(stream)))
    refs = dict(corr._keep)
    refs["records"] = out
    refs["perm"] = perm
    refs["src_ptr"] = refs["src_rec"] = None
    c2 = Corr.from_buffer_copy(c)
    c2.records = out.data_ptr()
    c2.mode = CORR_SPARSE
    c2.src_ptr = c2.src_rec = None  # the source index belongs to the unpermuted records
    return CorrHandle(c2, refs)


def raster_posmaps(verts, faces, face_off, cams, H, W, zbuf=None, pos=None, valid=None, stream=None, s=1):
    """geocache_raster_posmaps (s = 1) or geocache_raster_posmaps_supersampled
    (rendered at s times the token grid and pooled to it): position maps
    [B,N,H,W,3] f32 and validity [B,N,H,W] u8 of B meshes (verts [V,3] f32,
    faces [F,3] i32 indexing verts, face_off [B+1] i64, all on the device)
    seen by cams [B,N,16] (cameras of the H x W token grid).  Returns
    (pos, valid); zbuf is the [B,N,s*H,s*W] int64 scratch."""
    B, N = int(cams.shape[0]), int(cams.shape[1])
    dev = cams.device
    s = int(s)
    if zbuf is None:
        zbuf = torch.empty((B, N, s * H, s * W), dtype=torch.int64, device=dev)
    if pos is None:
        pos = torch.empty((B, N, H, W, 3), dtype=torch.float32, device=dev)
    if valid is None:
        valid = torch.empty((B, N, H, W), dtype=torch.uint8, device=dev)
    nv, nf = int(verts.shape[0]), int(faces.shape[0])
    n = B * N * H * W
    args = [_dev(verts, torch.float32, 3 * nv, "verts") if nv else None, nv,
            _dev(faces, torch.int32, 3 * nf, "faces") if nf else None, nf,
            _dev(face_off, torch.int64, B + 1, "face_off"), B, _dev(cams, torch.float32, 16 * B * N, "cams"), N,
            int(H), int(W)]
    outs = [_dev(zbuf, torch.int64, n * s * s, "zbuf"), _dev(pos, torch.float32, 3 * n, "pos"),
            _dev(valid, torch.uint8, n, "valid"), _stream(stream)]
    if s == 1:
        _check(load().geocache_raster_posmaps(*args, *outs))
    else:
        _check(load().geocache_raster_posmaps_supersampled(*args, s, *outs))
    return pos, valid


def pool_posmaps(pos_hi, valid_hi, s, pos=None, valid=None, stream=None):
    """geocache_pool_posmaps: token-grid maps ([..., H, W, 3] f32, [..., H, W]
    u8) from maps rendered at s times the token resolution (pos_hi [..., s*H,
    s*W, 3] f32, valid_hi [..., s*H, s*W] u8, on the device)."""
    s = int(s)
    Hs, Ws = int(valid_hi.shape[-2]), int(valid_hi.shape[-1])
    if Hs % s or Ws % s:
        raise ValueError("maps of %dx%d are not an s=%d super-sampling" % (Hs, Ws, s))
    H, W = Hs // s, Ws // s
    lead = tuple(valid_hi.shape[:-2])
    n_maps = 1
    for d in lead:
        n_maps *= int(d)
    if pos is None:
        pos = torch.empty(lead + (H, W, 3), dtype=torch.float32, device=valid_hi.device)
    if valid is None:
        valid = torch.empty(lead + (H, W), dtype=torch.uint8, device=valid_hi.device)
    n_hi, n = n_maps * Hs * Ws, n_maps * H * W
    _check(load().geocache_pool_posmaps(_dev(pos_hi, torch.float32, 3 * n_hi, "pos_hi"),
                                        _dev(valid_hi, torch.uint8, n_hi, "valid_hi"), n_maps, H, W, s,
                                        _dev(pos, torch.float32, 3 * n, "pos"), _dev(valid, torch.uint8, n, "valid"),
                                        _stream(stream)))
    return pos, valid


def transport_step_noalloc(corr: CorrHandle, anchors, C, x0_anchor_new, x0_prev, x0_out, x_t=None, x_next=None,
                           recon: Recon | None = None, stream=None):
    """geocache_transport_step_noalloc: the cached step for callers that
    cannot supply a workspace (the library's built-in scratch array is used;
    calls on one device must not overlap on the GPU)."""
    c = corr.c
    anc = sorted(int(a) for a in anchors)
    a = len(anc)
    n_all = c.B * c.N * C * c.H * c.W
    arr = (ctypes.c_int32 * max(1, a))(*anc)
    lat = F32
    pt = pn = None
    if recon is not None:
        lat = _lat_dtype(x_t)
        pt, pn = _dev(x_t, x_t.dtype, n_all, "x_t"), _dev(x_next, x_t.dtype, n_all, "x_next")
        _check_pred(recon, n_all)
    _check(load().geocache_transport_step_noalloc(
        ctypes.byref(c), ctypes.cast(arr, ctypes.c_void_p), a, int(C),
        _dev(x0_anchor_new, torch.float32, c.B * a * C * c.H * c.W, "x0_anchor_new"),
        _dev(x0_prev, torch.float32, n_all, "x0_prev"), _dev(x0_out, torch.float32, n_all, "x0_out"),
        pt, pn, lat, ctypes.byref(recon) if recon is not None else None, _stream(stream)))


def _rows(src_full, a):
    if src_full.dim() < 2:
        raise ValueError("per-view tensors are [B, N, ...]")
    B, N = src_full.shape[0], src_full.shape[1]
    return B, N, (src_full[0, 0].numel() if B * N else 0) * src_full.element_size()


def pack_anchors(src, dst, anchors, stream=None):
    """geocache_pack_anchors: dst [B, a, ...] <- src[:, anchors] (raw bytes)."""
    anc = sorted(int(x) for x in anchors)
    B, N, row = _rows(src, len(anc))
    if dst.dtype != src.dtype or tuple(dst.shape) != (B, len(anc)) + tuple(src.shape[2:]):
        raise ValueError("dst must be [B, a, ...] of src's dtype")
    arr = (ctypes.c_int32 * len(anc))(*anc)
    _check(load().geocache_pack_anchors(_dev(src, src.dtype, name="src"), _dev(dst, dst.dtype, name="dst"), row, B, N,
                                        ctypes.cast(arr, ctypes.c_void_p), len(anc), _stream(stream)))


def unpack_anchors(src, dst, anchors, stream=None):
    """geocache_unpack_anchors: dst[:, anchors] <- src [B, a, ...] (raw bytes)."""
    anc = sorted(int(x) for x in anchors)
    B, N, row = _rows(dst, len(anc))
    if src.dtype != dst.dtype or tuple(src.shape) != (B, len(anc)) + tuple(dst.shape[2:]):
        raise ValueError("src must be [B, a, ...] of dst's dtype")
    arr = (ctypes.c_int32 * len(anc))(*anc)
    _check(load().geocache_unpack_anchors(_dev(src, src.dtype, name="src"), _dev(dst, dst.dtype, name="dst"), row, B, N,
                                          ctypes.cast(arr, ctypes.c_void_p), len(anc), _stream(stream)))


def reconstruct(x_t, x0, x_next, recon: Recon, x0_store=None, stream=None):
    """geocache_reconstruct (full-step passthrough) on torch tensors."""
    n = x0.numel()
    dt = x_t.dtype
    _check_pred(recon, n)
    _check(load().geocache_reconstruct(_dev(x_t, dt, n, "x_t"), _dev(x0, torch.float32, n, "x0"),
                                       _dev(x_next, dt, n, "x_next"), _lat_dtype(x_t), n, ctypes.byref(recon),
                                       _dev(x0_store, torch.float32, n, "x0_store"), _stream(stream)))


def is_full_step(step: int, S: int, sched: dict) -> bool:
    s, _keep = make_schedule(sched)
    r = load().geocache_is_full_step(int(step), int(S), ctypes.byref(s))
    if r < 0:
        raise GeocacheError(r, last_error())
    return bool(r)


def rotate_anchors(N: int, a: int, step: int, S: int, sched: dict):
    """(anchors, is_full) of a step."""
    s, _keep = make_schedule(sched)
    out = (ctypes.c_int32 * a)()
    full = ctypes.c_int(0)
    _check(load().geocache_rotate_anchors(int(N), int(a), int(step), int(S), ctypes.byref(s),
                                          ctypes.cast(out, ctypes.c_void_p), ctypes.byref(full)))
    return list(out), bool(full.value)


def transport_launches(a: int, N: int, mode: int, in_place: bool = False) -> int:
    """Kernels one geocache_transport_step enqueues: sparse mode runs the
    record-parallel apply (when some view is outside the anchor set) and the
    streaming kernel; the other modes one fused kernel, plus the anchor-row
    copy of an in-place update."""
    if mode == CORR_SPARSE:
        return 2 if a < N else 1
    return 1 + (1 if in_place else 0)


def device_status(stream=None):
    """geocache_device_status (synchronises, reads and clears the device
    status word): raises GeocacheError with ESHAPE (a sparse build overflowed
    max_records), EINVAL (a record permutation entry or a mesh face index was
    out of range) or ETIMEOUT (a kernel's bounded wait gave up) for what
    happened since the last check."""
    _check(load().geocache_device_status(_stream(stream)))


def debug_set_wait(limit_ns: int = 0, drop_first_copy: bool = False):
    """geocache_debug_set_wait (test hook): limit of the kernels' bounded waits
    (0 = default), and whether the next staged transport call leaves its first
    unit's copies unissued so that its wait runs out."""
    _check(load().geocache_debug_set_wait(int(limit_ns), 1 if drop_first_copy else 0))


def abi_version() -> int:
    return load().geocache_abi_version()
