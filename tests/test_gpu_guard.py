"""Guard-band canaries: every output a kernel writes is placed inside a larger
buffer filled with a sentinel byte, and after the call the bytes before and
after the output must still hold it (no kernel writes outside its output's
extent).  Cases are chosen for the paths whose bounds are easiest to get
wrong: ragged token counts (H*W not a multiple of 4 or of the tile), channel
counts not a multiple of 4, pointers that are not 16-byte aligned (the
scalar paths), a record buffer filled exactly to capacity and one that
overflows, and the pooled and plain position maps."""
import numpy as np
import pytest
import torch

from paper_2608_13255_gb300 import synth

from gpu_helpers import step_inputs

pytestmark = pytest.mark.gpu

SENTINEL = 0xA5
PAD = 4096  # bytes of guard band on each side


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13255_gb300 import build as gbuild
    gbuild.build()
    from paper_2608_13255_gb300 import geocache
    geocache.load()
    return geocache


class Guarded:
    """A tensor of `shape` and `dtype` inside a sentinel-filled byte buffer,
    starting `skew` bytes after a 16-byte boundary."""

    def __init__(self, shape, dtype, skew=0, fill=None):
        n = int(np.prod(shape))
        self.nbytes = n * torch.tensor([], dtype=dtype).element_size()
        self.lo = PAD + skew
        self.buf = torch.full((PAD + skew + self.nbytes + PAD,), SENTINEL, dtype=torch.uint8, device="cuda")
        self.t = self.buf[self.lo:self.lo + self.nbytes].view(dtype).view(shape)
        if fill is not None:
            self.t.copy_(fill)

    def check(self, what):
        torch.cuda.synchronize()
        head = self.buf[:self.lo]
        tail = self.buf[self.lo + self.nbytes:]
        bad_h = int((head != SENTINEL).sum())
        bad_t = int((tail != SENTINEL).sum())
        assert bad_h == 0 and bad_t == 0, "%s: %d bytes before and %d bytes after the output were written" % (
            what, bad_h, bad_t)


def _geometry(gc, w, K=4, skew=0, records_frac=1.0):
    """tau, keep, tile_ptr, records and tables of w, each guarded."""
    dev = "cuda"
    pos, valid, cams = (torch.from_numpy(a).to(dev) for a in (w.pos, w.valid, w.cams))
    T = gc.tiles_per_view(w.H, w.W)
    # count with unguarded scratch first
    tau0 = torch.zeros(w.B, device=dev)
    keep0 = torch.empty((w.B, w.N, w.N, w.H, w.W), dtype=torch.uint8, device=dev)
    tp0 = torch.empty(w.B * w.N * w.N * T + 1, dtype=torch.int32, device=dev)
    R = gc.record_count(gc.make_corr(pos, valid, cams, tau0, K=K, keep=keep0, tile_ptr=tp0, mode=gc.CORR_MASK))
    cap = max(1, int(R * records_frac))
    g = {
        "tau": Guarded((w.B,), torch.float32, skew),
        "keep": Guarded((w.B, w.N, w.N, w.H, w.W), torch.uint8, skew + 1),
        "tile_ptr": Guarded((w.B * w.N * w.N * T + 1,), torch.int32, skew),
        "records": Guarded((cap, 4), torch.int32, 0),  # the ABI requires 16-byte aligned records
        "idx": Guarded((w.B, w.N, w.N, w.H, w.W, K), torch.int32, 0 if K == 4 else skew),
        "w": Guarded((w.B, w.N, w.N, w.H, w.W, K), torch.float32, 0 if K == 4 else skew),
        "src_ptr": Guarded((w.B * w.N * T + 1,), torch.int32, skew),
        "src_rec": Guarded((cap, 2), torch.int32, 0),  # 8-byte aligned
    }
    corr = gc.make_corr(pos, valid, cams, g["tau"].t, g["idx"].t, g["w"].t, K=K, keep=g["keep"].t,
                        tile_ptr=g["tile_ptr"].t, records=g["records"].t, mode=gc.CORR_SPARSE,
                        src_ptr=g["src_ptr"].t, src_rec=g["src_rec"].t)
    gc.build_corr(corr)
    torch.cuda.synchronize()
    return corr, g, R, cap, (pos, valid, cams)


@pytest.mark.parametrize("case", ["ragged_c5", "ragged_c18", "ragged_c18_src", "misaligned", "c3_k1"])
def test_transport_writes_only_its_outputs(gc, case):
    minimal_ws = False
    if case == "ragged_c5":  # 37 x 53 tokens: H*W = 1961, two tiles, a ragged quad; C = 5
        w, C, skew, K = synth.make_workload("batch128", B=2, H=37, W=53), 5, 0, 4
    elif case == "ragged_c18":  # the same with C = 18: the increment plane, a partial last channel group
        w, C, skew, K = synth.make_workload("batch128", B=2, H=37, W=53), 18, 0, 4
    elif case == "ragged_c18_src":  # C = 18 with the minimal workspace: the source-tile apply
        w, C, skew, K = synth.make_workload("batch128", B=2, H=37, W=53), 18, 0, 4
        minimal_ws = True
    elif case == "misaligned":  # 64 x 64 tokens, every buffer 4 bytes off a 16-byte boundary
        w, C, skew, K = synth.make_workload("hunyuan64"), 4, 4, 4
    else:
        w, C, skew, K = synth.make_workload("solids96", H=40, W=40), 3, 0, 1
    w = synth.Workload(**{**w.__dict__, "C": C})
    corr, g, R, cap, _ = _geometry(gc, w, K=K, skew=skew)
    for k, v in g.items():
        v.check("build: " + k)
    anchors = [0, 3]
    x0_prev, x0_new, xt32 = step_inputs(w, 3, anchors)
    shp = (w.B, w.N, C, w.H, w.W)
    lat = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    p = synth.recon_params(w, 5)
    pred_kind = "v" if p["sampler"] == "ddim" else "velocity"
    for mode in ("sparse", "mask", "table", "geometry"):
        m = {"sparse": gc.CORR_SPARSE, "mask": gc.CORR_MASK, "table": gc.CORR_TABLE, "geometry": gc.CORR_GEOMETRY}[mode]
        src = mode == "sparse"
        c2 = gc.make_corr(corr._keep["pos"], corr._keep["valid"], corr._keep["cams"], corr.tau, corr.idx, corr.w, K=K,
                          keep=corr.keep, tile_ptr=corr._keep["tile_ptr"], records=corr._keep["records"], mode=m,
                          src_ptr=corr._keep["src_ptr"] if src else None,
                          src_rec=corr._keep["src_rec"] if src else None)
        out = Guarded(shp, torch.float32, skew)
        xn = Guarded(shp, lat, skew)
        pred = Guarded(shp, torch.float32, skew)
        nws = c2.min_workspace_floats(C) if minimal_ws else c2.workspace_floats(C)
        ws = Guarded((max(nws, 4),), torch.float32, 0)
        r = gc.make_recon(p["sampler"], a_t=p.get("a_t", 0), a_prev=p.get("a_prev", 0), sigma=p.get("sigma", 0),
                          sigma_next=p.get("sigma_next", 0), pred_kind=pred_kind, pred_out=pred.t)
        d_prev = Guarded(shp, torch.float32, skew, torch.from_numpy(x0_prev))
        d_new = Guarded((w.B, len(anchors), C, w.H, w.W), torch.float32, skew, torch.from_numpy(x0_new))
        d_xt = Guarded(shp, lat, skew, torch.from_numpy(xt32).to(lat))
        gc.transport_step(c2, anchors, C, d_new.t, d_prev.t, out.t, d_xt.t, xn.t, r,
                          workspace=ws.t if mode == "sparse" else None)
        gc.device_status()
        for name, gb in (("x0_out", out), ("x_next", xn), ("pred", pred), ("workspace", ws), ("x0_prev", d_prev),
                         ("x0_new", d_new), ("x_t", d_xt)):
            gb.check("%s %s: %s" % (case, mode, name))
        assert torch.isfinite(out.t).all()
        # in place: x0_out = x0_prev and x_next = x_t
        if mode in ("sparse", "mask"):
            gc.transport_step(c2, anchors, C, d_new.t, d_prev.t, d_prev.t, d_xt.t, d_xt.t, r,
                              workspace=ws.t if mode == "sparse" else None)
            gc.device_status()
            d_prev.check("%s %s in place: x0" % (case, mode))
            d_xt.check("%s %s in place: x_t" % (case, mode))


@pytest.mark.parametrize("frac,C", [(1.0, 4), (0.5, 4), (1.0, 16), (0.5, 16)])
def test_record_buffer_at_and_beyond_capacity(gc, frac, C):
    # records filled exactly to max_records, and an overflowing build (half
    # the capacity needed): nothing is written past the buffer, the overflow
    # is reported, and a step over the truncated form stays inside its outputs
    # (C = 16: the increment-plane path)
    w = synth.make_workload("batch128", B=2, H=37, W=53)
    w = synth.Workload(**{**w.__dict__, "C": C})
    corr, g, R, cap, _ = _geometry(gc, w, K=4)
    if frac < 1.0:
        corr, g, R, cap, _ = _geometry(gc, w, K=4, records_frac=frac)
        with pytest.raises(gc.GeocacheError) as ei:
            gc.device_status()
        assert ei.value.status == gc.ESHAPE
    else:
        assert cap == R
        gc.device_status()
    for k, v in g.items():
        v.check("build (capacity %d of %d records): %s" % (cap, R, k))
    x0_prev, x0_new, _ = step_inputs(w, 3, [1, 4])
    shp = (w.B, w.N, w.C, w.H, w.W)
    out = Guarded(shp, torch.float32)
    ws = Guarded((corr.workspace_floats(w.C),), torch.float32)
    gc.transport_step(corr, [1, 4], w.C, torch.from_numpy(x0_new).cuda(), torch.from_numpy(x0_prev).cuda(), out.t,
                      workspace=ws.t)
    gc.device_status()
    out.check("step over %d of %d records: x0_out" % (cap, R))
    ws.check("step over %d of %d records: workspace" % (cap, R))


@pytest.mark.parametrize("s,H,W,skew", [(1, 37, 53, 4), (3, 20, 30, 0), (4, 16, 16, 4)])
def test_position_maps_write_only_their_outputs(gc, s, H, W, skew):
    rng = np.random.default_rng(5)
    V, F = synth.blob_mesh(3, 0.15, rng)
    cams = np.stack([synth.look_at_camera(az, el, H, W) for az, el in synth.hunyuan_layout()])[None]
    dev = "cuda"
    verts = torch.from_numpy(V.astype(np.float32)).to(dev)
    faces = torch.from_numpy(F.astype(np.int32)).to(dev)
    f_off = torch.tensor([0, len(F)], dtype=torch.int64, device=dev)
    d_cams = torch.from_numpy(cams.astype(np.float32)).to(dev)
    N = cams.shape[1]
    zb = Guarded((1, N, s * H, s * W), torch.int64, 0)
    pos = Guarded((1, N, H, W, 3), torch.float32, skew)
    valid = Guarded((1, N, H, W), torch.uint8, skew + 1)
    gc.raster_posmaps(verts, faces, f_off, d_cams, H, W, zb.t, pos.t, valid.t, s=s)
    gc.device_status()
    for name, gb in (("zbuf", zb), ("pos", pos), ("valid", valid)):
        gb.check("raster s=%d: %s" % (s, name))
    assert valid.t.float().mean() > 0.05
    # pooling caller-rendered fine maps
    fine_p = Guarded((1, N, s * H, s * W, 3), torch.float32, skew)
    fine_v = Guarded((1, N, s * H, s * W), torch.uint8, skew + 3)
    cams_hi = d_cams.clone()
    cams_hi[..., 12:16] *= s
    gc.raster_posmaps(verts, faces, f_off, cams_hi, s * H, s * W, zb.t, fine_p.t, fine_v.t)
    p2 = Guarded((1, N, H, W, 3), torch.float32, skew)
    v2 = Guarded((1, N, H, W), torch.uint8, skew + 2)
    gc.pool_posmaps(fine_p.t, fine_v.t, s, p2.t, v2.t)
    gc.device_status()
    p2.check("pool s=%d: pos" % s)
    v2.check("pool s=%d: valid" % s)
    assert torch.equal(v2.t, valid.t) and torch.equal(p2.t.view(torch.int32), pos.t.view(torch.int32))


def test_reconstruct_and_pack_write_only_their_outputs(gc):
    n = 4 * 1000 + 3  # not a multiple of 4
    x0 = torch.randn(n, device="cuda")
    for lat, skew in ((torch.bfloat16, 2), (torch.float32, 4), (torch.bfloat16, 0)):
        xt = torch.randn(n, device="cuda").to(lat)
        xn = Guarded((n,), lat, skew)
        fskew = 4 if skew else 0  # float outputs off a 16-byte boundary when the latents are
        pred = Guarded((n,), torch.float32, fskew)
        store = Guarded((n,), torch.float32, fskew)
        r = gc.make_recon("ddim", a_t=0.4, a_prev=0.5, pred_kind="eps", pred_out=pred.t)
        gc.reconstruct(xt, x0, xn.t, r, x0_store=store.t)
        gc.device_status()
        for name, gb in (("x_next", xn), ("pred", pred), ("x0_store", store)):
            gb.check("reconstruct %s skew %d: %s" % (lat, skew, name))
    # anchor-row pack / unpack with rows of 3 x 5 x 7 bf16 (210 bytes: 2-byte path)
    src = torch.randn((3, 6, 3, 5, 7), device="cuda").to(torch.bfloat16)
    dst = Guarded((3, 2, 3, 5, 7), torch.bfloat16, 2)
    gc.pack_anchors(src, dst.t, [1, 4])
    dst.check("pack")
    full = Guarded((3, 6, 3, 5, 7), torch.bfloat16, 2, src)
    gc.unpack_anchors(dst.t, full.t, [1, 4])
    full.check("unpack")
    assert torch.equal(full.t, src)
