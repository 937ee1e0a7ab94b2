// C ABI of libgeocache.so (include/geocache.h): argument checking, the host
// side of the anchor rotation and the refresh schedule, sampler constants,
// and kernel launches.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <string>

#include "geocache.h"
#include "geocache_internal.h"

namespace {

thread_local std::string g_last_error;

int fail(int status, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return status;
}

int ok() {
    g_last_error.clear();
    return GEOCACHE_OK;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(GEOCACHE_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// [a, a+na) and [b, b+nb) in bytes overlap
bool overlap(const void* a, size_t na, const void* b, size_t nb) {
    if (!a || !b || na == 0 || nb == 0) return false;
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return x < y + nb && y < x + na;
}

int check_sizes(int B, int N, int H, int W) {
    if (B < 1 || B > 65535) return fail(GEOCACHE_ESHAPE, "B=%d out of range [1, 65535]", B);
    if (N < 2 || N > GEOCACHE_MAX_VIEWS) return fail(GEOCACHE_ESHAPE, "N=%d out of range [2, %d]", N, GEOCACHE_MAX_VIEWS);
    if (H < 1 || W < 1 || H > 16384 || W > 16384) return fail(GEOCACHE_ESHAPE, "H=%d, W=%d out of range [1, 16384]", H, W);
    return GEOCACHE_OK;
}

int make_coef(const geocache_recon* r, geocache::ReconCoef* c) {
    *c = geocache::ReconCoef{};
    if (!r) return GEOCACHE_OK;
    c->enabled = 1;
    c->sampler = r->sampler;
    c->pred_kind = r->pred_kind;
    if (r->pred_kind != GEOCACHE_PRED_NONE && !r->pred_out)
        return fail(GEOCACHE_EINVAL, "pred_kind %d requires pred_out", (int)r->pred_kind);
    if (r->pred_kind == GEOCACHE_PRED_NONE && r->pred_out)
        return fail(GEOCACHE_EINVAL, "pred_out given with pred_kind NONE");
    if (r->sampler == GEOCACHE_DDIM) {
        if (!(r->a_t > 0.0 && r->a_t < 1.0)) return fail(GEOCACHE_EINVAL, "DDIM needs 0 < a_t < 1 (got %g)", r->a_t);
        if (!(r->a_prev > 0.0 && r->a_prev <= 1.0))
            return fail(GEOCACHE_EINVAL, "DDIM needs 0 < a_prev <= 1 (got %g)", r->a_prev);
        if (r->pred_kind != GEOCACHE_PRED_NONE && r->pred_kind != GEOCACHE_PRED_EPS && r->pred_kind != GEOCACHE_PRED_V)
            return fail(GEOCACHE_EINVAL, "DDIM prediction must be NONE, EPS or V");
        c->st = (float)std::sqrt(r->a_t);
        c->s1t = (float)std::sqrt(1.0 - r->a_t);
        c->inv_s1t = (float)(1.0 / std::sqrt(1.0 - r->a_t));
        c->sp = (float)std::sqrt(r->a_prev);
        c->s1p = (float)std::sqrt(1.0 - r->a_prev);
    } else if (r->sampler == GEOCACHE_FM_EULER) {
        if (!(r->sigma > 0.0 && std::isfinite(r->sigma)))
            return fail(GEOCACHE_EINVAL, "flow matching needs sigma > 0 (got %g)", r->sigma);
        if (!(r->sigma_next >= 0.0 && std::isfinite(r->sigma_next)))
            return fail(GEOCACHE_EINVAL, "flow matching needs sigma_next >= 0 (got %g)", r->sigma_next);
        if (r->pred_kind != GEOCACHE_PRED_NONE && r->pred_kind != GEOCACHE_PRED_VELOCITY)
            return fail(GEOCACHE_EINVAL, "flow-matching prediction must be NONE or VELOCITY");
        c->inv_sigma = (float)(1.0 / r->sigma);
        c->dsigma = (float)(r->sigma_next - r->sigma);
    } else {
        return fail(GEOCACHE_EINVAL, "unknown sampler %d", (int)r->sampler);
    }
    return GEOCACHE_OK;
}

size_t lat_bytes(int dtype) { return dtype == GEOCACHE_BF16 ? 2 : 4; }

// total record count of the sparse form (synchronises the stream)
int read_total(const geocache_corr* c, int64_t* total, cudaStream_t s) {
    const size_t n = (size_t)c->B * c->N * c->N * geocache::tiles_per_view(c->H, c->W);
    int32_t v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, c->tile_ptr + n, sizeof v, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "reading the record count");
    if (v < 0) return fail(GEOCACHE_ESHAPE, "the sparse form has more than 2^31-1 records");
    *total = v;
    return GEOCACHE_OK;
}

}  // namespace

int geocache::set_error(int status, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return status;
}

extern "C" {

int geocache_abi_version(void) { return GEOCACHE_ABI_VERSION; }

int geocache_device_status(void* stream) {
    unsigned int word = 0, raster_word = 0;
    cudaError_t e = geocache::read_device_error(&word, true, (cudaStream_t)stream);
    if (e == cudaSuccess) e = geocache::read_raster_error(&raster_word, true, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device status word");
    word |= raster_word;
    if (word & 2u)
        return fail(GEOCACHE_ESHAPE, "a sparse-form build had more records than max_records (status word 0x%x); "
                                     "query geocache_corr_record_count and rebuild", word);
    if (word & 4u)
        return fail(GEOCACHE_EINVAL, "a record permutation entry was outside [0, max_records) (status word 0x%x); "
                                     "those records were kept", word);
    if (word & 8u)
        return fail(GEOCACHE_EINVAL, "a mesh face had a vertex index outside [0, n_verts) (status word 0x%x); "
                                     "those faces were skipped", word);
    if (word & 16u)
        return fail(GEOCACHE_EINVAL, "a correspondence table index was outside [-1, H*W) (status word 0x%x); "
                                     "those taps were dropped", word);
    if (word) return fail(GEOCACHE_ETIMEOUT, "a bounded device wait gave up (status word 0x%x); outputs of that call are incomplete", word);
    return ok();
}

const char* geocache_last_error(void) { return g_last_error.c_str(); }

int geocache_debug_set_wait(uint64_t limit_ns, int drop_first_copy) {
    geocache::set_debug_wait((unsigned long long)limit_ns, drop_first_copy);
    return ok();
}

int geocache_build_corr(geocache_corr* c, void* stream) {
    if (!c) return fail(GEOCACHE_EINVAL, "corr is NULL");
    int st = check_sizes(c->B, c->N, c->H, c->W);
    if (st) return st;
    if (c->K != 1 && c->K != 4) return fail(GEOCACHE_EINVAL, "K=%d must be 1 or 4", c->K);
    if (!(c->tol_frac > 0.0f) || !std::isfinite(c->tol_frac))
        return fail(GEOCACHE_EINVAL, "tol_frac=%g must be positive", (double)c->tol_frac);
    if (!c->pos || !c->valid || !c->cams || !c->tau) return fail(GEOCACHE_EINVAL, "pos, valid, cams and tau are required");
    if ((c->idx == nullptr) != (c->w == nullptr)) return fail(GEOCACHE_EINVAL, "idx and w must both be given or both NULL");
    const size_t texels = (size_t)c->B * c->N * c->H * c->W;
    if (overlap(c->tau, sizeof(float) * c->B, c->pos, texels * 12) ||
        overlap(c->tau, sizeof(float) * c->B, c->valid, texels) ||
        overlap(c->tau, sizeof(float) * c->B, c->cams, sizeof(geocache_camera) * c->B * c->N))
        return fail(GEOCACHE_EALIAS, "tau overlaps an input");
    if (c->idx) {
        const size_t rows = texels * c->N * c->K;
        if (c->K == 4 && (((uintptr_t)c->idx | (uintptr_t)c->w) & 15))
            return fail(GEOCACHE_EINVAL, "idx and w must be 16-byte aligned for K=4");
        if (overlap(c->idx, rows * 4, c->w, rows * 4)) return fail(GEOCACHE_EALIAS, "idx and w overlap");
        if (c->keep && (overlap(c->keep, rows / c->K, c->idx, rows * 4) || overlap(c->keep, rows / c->K, c->w, rows * 4)))
            return fail(GEOCACHE_EALIAS, "keep overlaps idx or w");
    }
    if (c->keep && (overlap(c->keep, texels * c->N, c->pos, texels * 12) || overlap(c->keep, texels * c->N, c->valid, texels) ||
                    overlap(c->keep, texels * c->N, c->tau, sizeof(float) * c->B)))
        return fail(GEOCACHE_EALIAS, "keep overlaps an input");
    if (c->tile_ptr && !c->keep) return fail(GEOCACHE_EINVAL, "tile_ptr needs keep");
    if (c->records && !c->tile_ptr) return fail(GEOCACHE_EINVAL, "records need tile_ptr");
    if (c->records && (c->max_records < 0 || ((uintptr_t)c->records & 15)))
        return fail(GEOCACHE_EINVAL, "records must be 16-byte aligned with max_records >= 0");
    if (c->tile_ptr) {
        const size_t nt = (size_t)c->B * c->N * c->N * geocache::tiles_per_view(c->H, c->W) + 1;
        if (overlap(c->tile_ptr, nt * 4, c->keep, texels * c->N) || overlap(c->tile_ptr, nt * 4, c->pos, texels * 12) ||
            (c->records && overlap(c->tile_ptr, nt * 4, c->records, (size_t)c->max_records * 16)))
            return fail(GEOCACHE_EALIAS, "tile_ptr overlaps another buffer");
    }
    if (c->records && (overlap(c->records, (size_t)c->max_records * 16, c->pos, texels * 12) ||
                       overlap(c->records, (size_t)c->max_records * 16, c->keep, texels * c->N)))
        return fail(GEOCACHE_EALIAS, "records overlap another buffer");
    if ((c->src_ptr == nullptr) != (c->src_rec == nullptr))
        return fail(GEOCACHE_EINVAL, "src_ptr and src_rec must both be given or both NULL");
    if (c->src_ptr) {
        if (!c->records) return fail(GEOCACHE_EINVAL, "the source index needs records");
        if ((uintptr_t)c->src_rec & 7) return fail(GEOCACHE_EINVAL, "src_rec must be 8-byte aligned");
        const size_t ng = ((size_t)c->B * c->N * geocache::tiles_per_view(c->H, c->W) + 1) * 4;
        const size_t nr = (size_t)c->max_records * 8, nt = ((size_t)c->B * c->N * c->N * geocache::tiles_per_view(c->H, c->W) + 1) * 4;
        const void* bufs[4] = {c->records, c->tile_ptr, c->keep, c->pos};
        const size_t sizes[4] = {(size_t)c->max_records * 16, nt, texels * c->N, texels * 12};
        if (overlap(c->src_ptr, ng, c->src_rec, nr)) return fail(GEOCACHE_EALIAS, "src_ptr and src_rec overlap");
        for (int i = 0; i < 4; ++i)
            if (overlap(c->src_ptr, ng, bufs[i], sizes[i]) || overlap(c->src_rec, nr, bufs[i], sizes[i]))
                return fail(GEOCACHE_EALIAS, "the source index overlaps another buffer");
    }
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = geocache::launch_tau(c->pos, c->valid, c->B, c->N, c->H, c->W, c->tol_frac, c->tau, s);
    if (e != cudaSuccess) return cuda_fail(e, "tau kernel launch");
    if (c->idx || c->keep) {
        e = geocache::launch_build_corr(*c, s);
        if (e != cudaSuccess) return cuda_fail(e, "correspondence kernel launch");
    }
    if (c->tile_ptr) {
        e = geocache::launch_tile_ptr(*c, s);
        if (e != cudaSuccess) return cuda_fail(e, "tile-offset kernel launch");
    }
    if (c->records) {
        e = geocache::launch_fill_records(*c, s);
        if (e != cudaSuccess) return cuda_fail(e, "record kernel launch");
    }
    if (c->src_ptr) {
        e = geocache::launch_src_index(*c, s);
        if (e != cudaSuccess) return cuda_fail(e, "source index kernel launch");
    }
    return ok();
}

int geocache_corr_record_count(geocache_corr* c, int64_t* count, void* stream) {
    if (!c || !count) return fail(GEOCACHE_EINVAL, "corr and count are required");
    if (!c->keep || !c->tile_ptr) return fail(GEOCACHE_EINVAL, "counting records needs keep and tile_ptr");
    geocache_corr d = *c;
    d.records = nullptr;
    d.src_ptr = nullptr;
    d.src_rec = nullptr;
    d.idx = nullptr;
    d.w = nullptr;
    int st = geocache_build_corr(&d, stream);
    if (st) return st;
    return read_total(c, count, (cudaStream_t)stream);
}

int64_t geocache_transport_workspace(const geocache_corr* c, int C) {
    if (!c || C < 1 || c->mode != GEOCACHE_CORR_SPARSE || c->max_records < 0) return 0;
    int64_t n = c->max_records * (int64_t)C;
    // room for the anchors' increment plane of any step with a < N
    if (C >= geocache::kPlaneMinChannels && c->N > 1)
        n += geocache::plane_floats(c->B, c->N - 1, C, (long long)c->H * c->W);
    return n;
}

int geocache_transport_step(const geocache_corr* c, const int32_t* anchors, int a, int C,
                            const float* x0_anchor_new, const float* x0_prev, float* x0_out, const void* x_t,
                            void* x_next, geocache_dtype lat_dtype, const geocache_recon* recon, float* workspace,
                            int64_t workspace_floats, void* stream) {
    return geocache_transport_step_update(c, GEOCACHE_UPDATE_DELTA, anchors, a, C, x0_anchor_new, x0_prev, x0_out,
                                          x_t, x_next, lat_dtype, recon, workspace, workspace_floats, stream);
}

int geocache_transport_step_update(const geocache_corr* c, geocache_update update, const int32_t* anchors, int a,
                                   int C, const float* x0_anchor_new, const float* x0_prev, float* x0_out,
                                   const void* x_t, void* x_next, geocache_dtype lat_dtype,
                                   const geocache_recon* recon, float* workspace, int64_t workspace_floats,
                                   void* stream) {
    if (!c) return fail(GEOCACHE_EINVAL, "corr is NULL");
    if (update != GEOCACHE_UPDATE_DELTA && update != GEOCACHE_UPDATE_COPY)
        return fail(GEOCACHE_EINVAL, "unknown update rule %d", (int)update);
    int st = check_sizes(c->B, c->N, c->H, c->W);
    if (st) return st;
    if (c->K != 1 && c->K != 4) return fail(GEOCACHE_EINVAL, "K=%d must be 1 or 4", c->K);
    if (C < 1 || C > GEOCACHE_MAX_CHANNELS) return fail(GEOCACHE_ESHAPE, "C=%d out of range [1, %d]", C, GEOCACHE_MAX_CHANNELS);
    if (c->mode == GEOCACHE_CORR_GEOMETRY) {
        if (!c->pos || !c->valid || !c->cams || !c->tau)
            return fail(GEOCACHE_EINVAL, "geometry mode needs pos, valid, cams and tau");
    } else if (c->mode == GEOCACHE_CORR_TABLE) {
        if (!c->idx || !c->w) return fail(GEOCACHE_EINVAL, "table mode needs idx and w");
    } else if (c->mode == GEOCACHE_CORR_MASK) {
        if (!c->keep || !c->pos || !c->valid || !c->cams || !c->tau)
            return fail(GEOCACHE_EINVAL, "mask mode needs keep, pos, valid, cams and tau");
    } else if (c->mode == GEOCACHE_CORR_SPARSE) {
        if (!c->tile_ptr || !c->records || ((uintptr_t)c->records & 15))
            return fail(GEOCACHE_EINVAL, "sparse mode needs tile_ptr and 16-byte aligned records");
        if (a < c->N && (!workspace || workspace_floats < c->max_records * (int64_t)C))
            return fail(GEOCACHE_EINVAL, "sparse mode needs a workspace of max_records * C = %lld floats",
                        (long long)(c->max_records * (int64_t)C));
        if (((uintptr_t)workspace & 15)) return fail(GEOCACHE_EINVAL, "workspace must be 16-byte aligned");
    } else {
        return fail(GEOCACHE_EINVAL, "unknown corr mode %d", (int)c->mode);
    }
    if (!anchors) return fail(GEOCACHE_EINVAL, "anchors is NULL");
    if (a < 1 || a > c->N) return fail(GEOCACHE_EINVAL, "a=%d must be in [1, N=%d]", a, c->N);
    for (int s = 0; s < a; ++s) {
        if (anchors[s] < 0 || anchors[s] >= c->N) return fail(GEOCACHE_EINVAL, "anchor %d out of range", anchors[s]);
        if (s && anchors[s] <= anchors[s - 1]) return fail(GEOCACHE_EINVAL, "anchors must be ascending and distinct");
    }
    if (!x0_anchor_new || !x0_prev || !x0_out) return fail(GEOCACHE_EINVAL, "x0 buffers are required");
    if (lat_dtype != GEOCACHE_F32 && lat_dtype != GEOCACHE_BF16)
        return fail(GEOCACHE_EDTYPE, "unsupported latent dtype %d", (int)lat_dtype);
    geocache::ReconCoef coef;
    st = make_coef(recon, &coef);
    if (st) return st;
    const size_t HW = (size_t)c->H * c->W;
    const size_t n_all = (size_t)c->B * c->N * C * HW, n_anc = (size_t)c->B * a * C * HW;
    if (recon && (!x_t || !x_next)) return fail(GEOCACHE_EINVAL, "reconstruction needs x_t and x_next");
    if (x0_out != x0_prev && overlap(x0_out, n_all * 4, x0_prev, n_all * 4))
        return fail(GEOCACHE_EALIAS, "x0_out partially overlaps x0_prev");
    if (overlap(x0_out, n_all * 4, x0_anchor_new, n_anc * 4)) return fail(GEOCACHE_EALIAS, "x0_out overlaps x0_anchor_new");
    if (recon) {
        const size_t lb = lat_bytes(lat_dtype);
        if (x_next != x_t && overlap(x_next, n_all * lb, x_t, n_all * lb))
            return fail(GEOCACHE_EALIAS, "x_next partially overlaps x_t");
        if (overlap(x_next, n_all * lb, x0_out, n_all * 4) || overlap(x_next, n_all * lb, x0_prev, n_all * 4) ||
            overlap(x_next, n_all * lb, x0_anchor_new, n_anc * 4))
            return fail(GEOCACHE_EALIAS, "x_next overlaps an x0 buffer");
        if (recon->pred_out &&
            (overlap(recon->pred_out, n_all * 4, x0_out, n_all * 4) || overlap(recon->pred_out, n_all * 4, x_next, n_all * lb) ||
             overlap(recon->pred_out, n_all * 4, x0_prev, n_all * 4) || overlap(recon->pred_out, n_all * 4, x_t, n_all * lb)))
            return fail(GEOCACHE_EALIAS, "pred_out overlaps another buffer");
    }
    if (c->mode == GEOCACHE_CORR_SPARSE && workspace) {
        const size_t wb = (size_t)workspace_floats * 4, lb = lat_bytes(lat_dtype);
        if (overlap(workspace, wb, x0_out, n_all * 4) || overlap(workspace, wb, x0_prev, n_all * 4) ||
            overlap(workspace, wb, x0_anchor_new, n_anc * 4) ||
            (recon && (overlap(workspace, wb, x_next, n_all * lb) || overlap(workspace, wb, x_t, n_all * lb))))
            return fail(GEOCACHE_EALIAS, "workspace overlaps another buffer");
    }
    geocache::TransportArgs t{};
    t.B = c->B; t.N = c->N; t.H = c->H; t.W = c->W; t.C = C; t.K = c->K; t.a = a;
    t.mode = c->mode;
    // the sparse mode gathers in a kernel that completes before any row is
    // written, so an in-place update needs no separate anchor-row pass
    t.write_anchor_rows = (x0_out != x0_prev) || c->mode == GEOCACHE_CORR_SPARSE;
    t.lat_dtype = lat_dtype;
    t.update = update;
    t.pos = c->pos; t.valid = c->valid; t.cams = c->cams; t.tau = c->tau; t.idx = c->idx; t.w = c->w;
    t.keep = c->keep;
    t.tile_ptr = c->tile_ptr;
    t.records = c->records;
    t.max_records = c->max_records;
    t.src_ptr = c->mode == GEOCACHE_CORR_SPARSE ? c->src_ptr : nullptr;
    t.src_rec = c->mode == GEOCACHE_CORR_SPARSE ? c->src_rec : nullptr;
    t.workspace = workspace;
    t.workspace_floats = workspace ? workspace_floats : 0;
    t.x0_new = x0_anchor_new; t.x0_prev = x0_prev; t.x0_out = x0_out;
    t.x_t = x_t; t.x_next = x_next; t.pred_out = recon ? recon->pred_out : nullptr;
    t.coef = coef;
    for (int v = 0; v < GEOCACHE_MAX_VIEWS; ++v) { t.slot_of[v] = -1; t.anchors[v] = -1; t.others[v] = -1; }
    for (int s = 0; s < a; ++s) { t.anchors[s] = anchors[s]; t.slot_of[anchors[s]] = s; }
    for (int v = 0, k = 0; v < c->N; ++v)
        if (t.slot_of[v] < 0) t.others[k++] = v;
    cudaStream_t s = (cudaStream_t)stream;
    t.c0 = 0;
    t.cn = C;
    cudaError_t e = geocache::launch_transport(t, s);
    if (e != cudaSuccess) return cuda_fail(e, "transport kernel launch");
    if (!t.write_anchor_rows) {
        e = geocache::launch_copy_anchor_rows(t, s);
        if (e != cudaSuccess) return cuda_fail(e, "anchor-row copy launch");
    }
    return ok();
}

int geocache_permute_records(const geocache_corr* c, const int32_t* perm, geocache_tap_record* out, void* stream) {
    if (!c || !perm || !out) return fail(GEOCACHE_EINVAL, "corr, perm and out are required");
    if (!c->records || c->max_records < 0) return fail(GEOCACHE_EINVAL, "corr has no sparse records");
    if (((uintptr_t)out | (uintptr_t)c->records) & 15) return fail(GEOCACHE_EINVAL, "records must be 16-byte aligned");
    const size_t rb = (size_t)c->max_records * 16, pb = (size_t)c->max_records * 4;
    if (overlap(out, rb, c->records, rb) || overlap(out, rb, perm, pb))
        return fail(GEOCACHE_EALIAS, "out overlaps the records or the permutation");
    cudaError_t e = geocache::launch_permute_records(c->records, perm, out, c->max_records, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "record permutation kernel launch");
    return ok();
}

static int raster_entry(const char* fn, const float* verts, int64_t n_verts, const int32_t* faces, int64_t n_faces,
                        const int64_t* face_off, int B, const geocache_camera* cams, int N, int H, int W, int ss,
                        uint64_t* zbuf, float* pos, uint8_t* valid, void* stream) {
    if (B < 1 || B > 65535 || N < 1 || N > GEOCACHE_MAX_VIEWS || H < 1 || W < 1 || H > 16384 || W > 16384)
        return fail(GEOCACHE_ESHAPE, "%s: B=%d, N=%d, H=%d, W=%d out of range", fn, B, N, H, W);
    if (ss < 1 || ss > 16 || (int64_t)H * ss > 16384 || (int64_t)W * ss > 16384)
        return fail(GEOCACHE_ESHAPE, "%s: s=%d out of range (1 <= s <= 16, s*H and s*W <= 16384)", fn, ss);
    if (n_verts < 0 || n_faces < 0 || n_faces > 0xffffffffLL || n_verts > 0x7fffffffLL)
        return fail(GEOCACHE_ESHAPE, "%s: n_verts=%lld, n_faces=%lld out of range", fn, (long long)n_verts,
                    (long long)n_faces);
    if (!cams || !face_off || !zbuf || !pos || !valid || (n_faces > 0 && (!verts || !faces)))
        return fail(GEOCACHE_EINVAL, "%s: verts, faces, face_off, cams, zbuf, pos and valid are required", fn);
    if ((uintptr_t)zbuf & 7) return fail(GEOCACHE_EINVAL, "%s: zbuf must be 8-byte aligned", fn);
    const size_t px = (size_t)B * N * H * W;
    const void* outs[3] = {zbuf, pos, valid};
    const size_t ob[3] = {px * ss * ss * 8, px * 12, px};
    const void* ins[5] = {verts, faces, face_off, cams, nullptr};
    const size_t ib[5] = {(size_t)n_verts * 12, (size_t)n_faces * 12, (size_t)(B + 1) * 8, sizeof(geocache_camera) * B * N, 0};
    for (int i = 0; i < 3; ++i) {
        for (int j = i + 1; j < 3; ++j)
            if (overlap(outs[i], ob[i], outs[j], ob[j])) return fail(GEOCACHE_EALIAS, "%s: zbuf, pos and valid overlap", fn);
        for (int j = 0; j < 4; ++j)
            if (overlap(outs[i], ob[i], ins[j], ib[j])) return fail(GEOCACHE_EALIAS, "%s: an output overlaps an input", fn);
    }
    cudaError_t e = geocache::launch_raster(verts, n_verts, faces, n_faces, face_off, B, cams, N, H, W, ss,
                                            reinterpret_cast<unsigned long long*>(zbuf), pos, valid,
                                            (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

int geocache_raster_posmaps(const float* verts, int64_t n_verts, const int32_t* faces, int64_t n_faces,
                            const int64_t* face_off, int B, const geocache_camera* cams, int N, int H, int W,
                            uint64_t* zbuf, float* pos, uint8_t* valid, void* stream) {
    return raster_entry("geocache_raster_posmaps", verts, n_verts, faces, n_faces, face_off, B, cams, N, H, W, 1, zbuf,
                        pos, valid, stream);
}

int geocache_raster_posmaps_supersampled(const float* verts, int64_t n_verts, const int32_t* faces, int64_t n_faces,
                                         const int64_t* face_off, int B, const geocache_camera* cams, int N, int H,
                                         int W, int s, uint64_t* zbuf, float* pos, uint8_t* valid, void* stream) {
    return raster_entry("geocache_raster_posmaps_supersampled", verts, n_verts, faces, n_faces, face_off, B, cams, N,
                        H, W, s, zbuf, pos, valid, stream);
}

int geocache_pool_posmaps(const float* pos_hi, const uint8_t* valid_hi, int64_t n_maps, int H, int W, int s, float* pos,
                          uint8_t* valid, void* stream) {
    if (n_maps < 0 || H < 1 || W < 1 || H > 16384 || W > 16384)
        return fail(GEOCACHE_ESHAPE, "geocache_pool_posmaps: n_maps=%lld, H=%d, W=%d out of range", (long long)n_maps, H, W);
    if (s < 1 || s > 16 || (int64_t)H * s > 16384 || (int64_t)W * s > 16384)
        return fail(GEOCACHE_ESHAPE, "geocache_pool_posmaps: s=%d out of range (1 <= s <= 16, s*H and s*W <= 16384)", s);
    if (n_maps > 0 && (!pos_hi || !valid_hi || !pos || !valid))
        return fail(GEOCACHE_EINVAL, "geocache_pool_posmaps: pos_hi, valid_hi, pos and valid are required");
    const size_t tok = (size_t)n_maps * H * W, fine = tok * s * s;
    if (overlap(pos, tok * 12, pos_hi, fine * 12) || overlap(pos, tok * 12, valid_hi, fine) ||
        overlap(valid, tok, pos_hi, fine * 12) || overlap(valid, tok, valid_hi, fine) || overlap(pos, tok * 12, valid, tok))
        return fail(GEOCACHE_EALIAS, "geocache_pool_posmaps: an output overlaps an input or the other output");
    cudaError_t e = geocache::launch_pool_posmaps(pos_hi, valid_hi, n_maps, H, W, s, pos, valid, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "geocache_pool_posmaps");
    return ok();
}

int geocache_reconstruct(const void* x_t, const float* x0, void* x_next, geocache_dtype lat_dtype, int64_t n,
                         const geocache_recon* recon, float* x0_store, void* stream) {
    if (n < 0) return fail(GEOCACHE_ESHAPE, "n=%lld is negative", (long long)n);
    if (!recon) return fail(GEOCACHE_EINVAL, "recon is NULL");
    if (lat_dtype != GEOCACHE_F32 && lat_dtype != GEOCACHE_BF16)
        return fail(GEOCACHE_EDTYPE, "unsupported latent dtype %d", (int)lat_dtype);
    if (n > 0 && (!x_t || !x0 || !x_next)) return fail(GEOCACHE_EINVAL, "x_t, x0 and x_next are required");
    geocache::ReconCoef coef;
    int st = make_coef(recon, &coef);
    if (st) return st;
    const size_t lb = lat_bytes(lat_dtype), un = (size_t)n;
    if (x_next != x_t && overlap(x_next, un * lb, x_t, un * lb))
        return fail(GEOCACHE_EALIAS, "x_next partially overlaps x_t");
    if (overlap(x_next, un * lb, x0, un * 4)) return fail(GEOCACHE_EALIAS, "x_next overlaps x0");
    if (x0_store && x0_store != x0 &&
        (overlap(x0_store, un * 4, x0, un * 4) || overlap(x0_store, un * 4, x_next, un * lb) ||
         overlap(x0_store, un * 4, x_t, un * lb)))
        return fail(GEOCACHE_EALIAS, "x0_store overlaps another buffer");
    if (recon->pred_out && (overlap(recon->pred_out, un * 4, x_next, un * lb) || overlap(recon->pred_out, un * 4, x0, un * 4) ||
                            overlap(recon->pred_out, un * 4, x_t, un * lb)))
        return fail(GEOCACHE_EALIAS, "pred_out overlaps another buffer");
    cudaError_t e = geocache::launch_reconstruct(x_t, x0, x_next, lat_dtype, n, coef, recon->pred_out,
                                                 x0_store == x0 ? nullptr : x0_store, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "reconstruction kernel launch");
    return ok();
}

static int copy_rows_entry(const void* src, void* dst, int64_t row_bytes, int B, int N, const int32_t* anchors, int a,
                           bool pack, void* stream) {
    const char* fn = pack ? "geocache_pack_anchors" : "geocache_unpack_anchors";
    if (B < 0 || B > 65535) return fail(GEOCACHE_ESHAPE, "%s: B=%d out of range [0, 65535]", fn, B);
    if (N < 1 || N > GEOCACHE_MAX_VIEWS) return fail(GEOCACHE_ESHAPE, "%s: N=%d out of range [1, %d]", fn, N, GEOCACHE_MAX_VIEWS);
    if (row_bytes < 0) return fail(GEOCACHE_ESHAPE, "%s: row_bytes=%lld is negative", fn, (long long)row_bytes);
    if (!anchors) return fail(GEOCACHE_EINVAL, "%s: anchors is NULL", fn);
    if (a < 1 || a > N) return fail(GEOCACHE_EINVAL, "%s: a=%d must be in [1, N=%d]", fn, a, N);
    geocache::RowAnchors anc{};
    for (int s2 = 0; s2 < a; ++s2) {
        if (anchors[s2] < 0 || anchors[s2] >= N) return fail(GEOCACHE_EINVAL, "%s: anchor %d out of range", fn, anchors[s2]);
        if (s2 && anchors[s2] <= anchors[s2 - 1])
            return fail(GEOCACHE_EINVAL, "%s: anchors must be ascending and distinct", fn);
        anc.v[s2] = anchors[s2];
    }
    const size_t full = (size_t)B * N * (size_t)row_bytes, part = (size_t)B * a * (size_t)row_bytes;
    if (full && (!src || !dst)) return fail(GEOCACHE_EINVAL, "%s: src and dst are required", fn);
    if (overlap(src, pack ? full : part, dst, pack ? part : full))
        return fail(GEOCACHE_EALIAS, "%s: src and dst overlap", fn);
    cudaError_t e = geocache::launch_copy_rows(src, dst, row_bytes, B, N, a, anc, pack, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
}

int geocache_pack_anchors(const void* src, void* dst, int64_t row_bytes, int B, int N, const int32_t* anchors, int a,
                          void* stream) {
    return copy_rows_entry(src, dst, row_bytes, B, N, anchors, a, true, stream);
}

int geocache_unpack_anchors(const void* src, void* dst, int64_t row_bytes, int B, int N, const int32_t* anchors,
                            int a, void* stream) {
    return copy_rows_entry(src, dst, row_bytes, B, N, anchors, a, false, stream);
}

int geocache_is_full_step(int step, int S, const geocache_schedule* sched) {
    if (!sched) return fail(GEOCACHE_EINVAL, "schedule is NULL");
    if (S < 1 || step < 0 || step >= S) return fail(GEOCACHE_ESHAPE, "step=%d outside [0, S=%d)", step, S);
    switch (sched->kind) {
        case GEOCACHE_SCHED_SINGLE_CACHED:
            g_last_error.clear();
            return step == 0 ? 1 : 0;
        case GEOCACHE_SCHED_EVERY_K:
            if (sched->k < 1) return fail(GEOCACHE_EINVAL, "every-k schedule needs k >= 1");
            g_last_error.clear();
            return step % sched->k == 0 ? 1 : 0;
        case GEOCACHE_SCHED_HEAD_MID_TAIL:
            if (sched->head < 0 || sched->tail < 0) return fail(GEOCACHE_EINVAL, "head and tail must be >= 0");
            g_last_error.clear();
            if (step == 0 || step < sched->head) return 1;
            if (sched->mid && step == S / 2) return 1;
            return step >= S - sched->tail ? 1 : 0;
        case GEOCACHE_SCHED_LIST:
            if (sched->n_full_steps < 0 || (sched->n_full_steps > 0 && !sched->full_steps))
                return fail(GEOCACHE_EINVAL, "list schedule needs full_steps");
            g_last_error.clear();
            if (step == 0) return 1;
            for (int i = 0; i < sched->n_full_steps; ++i)
                if (sched->full_steps[i] == step) return 1;
            return 0;
        case GEOCACHE_SCHED_ALL_FULL:
            g_last_error.clear();
            return 1;
    }
    return fail(GEOCACHE_EINVAL, "unknown schedule kind %d", (int)sched->kind);
}

int geocache_rotate_anchors(int N, int a, int step, int S, const geocache_schedule* sched, int32_t* anchors_out,
                            int* is_full_out) {
    if (!anchors_out) return fail(GEOCACHE_EINVAL, "anchors_out is NULL");
    if (N < 1 || N > GEOCACHE_MAX_VIEWS) return fail(GEOCACHE_ESHAPE, "N=%d out of range [1, %d]", N, GEOCACHE_MAX_VIEWS);
    if (a < 1 || a > N) return fail(GEOCACHE_EINVAL, "a=%d must be in [1, N=%d]", a, N);
    int full = geocache_is_full_step(step, S, sched);
    if (full < 0) return full;
    int ordinal = 0;
    for (int t = 0; t < step; ++t) {
        const int f = geocache_is_full_step(t, S, sched);
        if (f < 0) return f;
        ordinal += f ? 0 : 1;
    }
    int cand[GEOCACHE_MAX_VIEWS];
    if (sched->contiguous_rotation) {
        for (int j = 0; j < a; ++j) cand[j] = (int)(((long long)ordinal * a + j) % N);
    } else {
        const int s = (N + a - 1) / a;
        const int r = ordinal % s;
        for (int j = 0; j < a; ++j) cand[j] = (r + j * s) % N;
    }
    bool used[GEOCACHE_MAX_VIEWS] = {false};
    bool in_cand[GEOCACHE_MAX_VIEWS] = {false};
    for (int j = 0; j < a; ++j) in_cand[cand[j]] = true;
    int out[GEOCACHE_MAX_VIEWS];
    for (int j = 0; j < a; ++j) {
        int x = cand[j];
        if (used[x]) {
            x = -1;
            for (int y = 0; y < N; ++y)
                if (!used[y] && !in_cand[y]) { x = y; break; }
            if (x < 0)
                for (int y = 0; y < N; ++y)
                    if (!used[y]) { x = y; break; }
        }
        used[x] = true;
        out[j] = x;
    }
    // ascending order
    for (int i = 1; i < a; ++i)
        for (int j = i; j > 0 && out[j - 1] > out[j]; --j) { int tmp = out[j]; out[j] = out[j - 1]; out[j - 1] = tmp; }
    for (int j = 0; j < a; ++j) anchors_out[j] = out[j];
    if (is_full_out) *is_full_out = full;
    return ok();
}

}  // extern "C"
