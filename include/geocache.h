/*
 * geocache.h -- C ABI of libgeocache.so: geometric delta transport between the
 * views of a multi-view diffusion batch (GeoCache, Sec. 3.2 of the paper),
 * computed by CUDA kernels for sm_103a on one GPU.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Pointers marked "device" are CUDA device addresses on the current device
 *   (e.g. torch tensors' data_ptr()); pointers marked "host" are ordinary host
 *   memory.  The caller owns every buffer and the library allocates no
 *   memory; its device-resident state is a 4-byte status word that kernels
 *   set on a failure they can only detect on the GPU (geocache_device_status)
 *   and the fixed scratch array of geocache_transport_step_noalloc.
 * - Every device-side entry point is asynchronous on `stream` (a cudaStream_t,
 *   NULL = the legacy default stream) and returns after enqueueing its kernels.
 * - Latents are NCHW per view with the views on the batch axis:
 *   [B, N, C, H, W] contiguous (B assets, N views, C channels, H x W tokens).
 *   Position maps and correspondence tables use the same token grid.
 * - Arguments are checked before anything is launched; a non-OK status means
 *   nothing was enqueued (except GEOCACHE_ECUDA, which reports a launch
 *   failure after enqueueing) and geocache_last_error() describes the problem.
 */
#ifndef GEOCACHE_H
#define GEOCACHE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GEOCACHE_ABI_VERSION 2
#define GEOCACHE_MAX_VIEWS 64   /* N <= 64 */
#define GEOCACHE_MAX_CHANNELS 1024
#define GEOCACHE_TILE_TOKENS 1024 /* tokens per tile of the sparse operator (row-major token order) */

typedef enum {
    GEOCACHE_OK = 0,
    GEOCACHE_EINVAL = -1,   /* NULL pointer, bad enum, bad anchors, bad sampler parameters */
    GEOCACHE_ESHAPE = -2,   /* a size is out of range */
    GEOCACHE_EDTYPE = -3,   /* unsupported latent dtype */
    GEOCACHE_ECUDA = -4,    /* a CUDA call or kernel launch failed */
    GEOCACHE_ETIMEOUT = -5, /* a bounded device wait gave up (see geocache_device_status) */
    GEOCACHE_EDEVICE = -6,  /* no usable CUDA device */
    GEOCACHE_EALIAS = -7    /* buffers overlap in a way the call does not allow */
} geocache_status;

typedef enum { GEOCACHE_F32 = 0, GEOCACHE_BF16 = 1 } geocache_dtype;

typedef enum { GEOCACHE_DDIM = 0, GEOCACHE_FM_EULER = 1 } geocache_sampler;

/* Optional per-element prediction written next to x_{t-1}: the quantity a
 * sampler keeps in its history (Sec. 3.2, closed-form conversion after Eq. 1). */
typedef enum {
    GEOCACHE_PRED_NONE = 0,
    GEOCACHE_PRED_EPS = 1,      /* DDIM: eps = (x_t - sqrt(ab_t) x0) / sqrt(1 - ab_t) */
    GEOCACHE_PRED_V = 2,        /* DDIM: v = sqrt(ab_t) eps - sqrt(1 - ab_t) x0 */
    GEOCACHE_PRED_VELOCITY = 3  /* FM: u = (x_sigma - x0) / sigma */
} geocache_pred;

/* How geocache_transport_step obtains the taps of G_{u->v}.  All four give
 * bit-identical taps, weights and results. */
typedef enum {
    GEOCACHE_CORR_GEOMETRY = 0, /* recompute every tap test from pos/valid/cams/tau */
    GEOCACHE_CORR_TABLE = 1,    /* read idx/w written by geocache_build_corr (or supplied by the caller) */
    GEOCACHE_CORR_MASK = 2,     /* read the 1-byte keep masks written by geocache_build_corr; recompute
                                   the projection and weights only where a tap is kept */
    GEOCACHE_CORR_SPARSE = 3    /* read the sparse tap records written by geocache_build_corr (fastest):
                                   C < 8, or a workspace without room for the increment plane: the
                                   records are applied record-parallel (or per source tile with a
                                   source index) into workspace rows; C >= 8 with room: the anchors'
                                   increments are written as a plane and gathered per record */
} geocache_corr_mode;

/* Update rule of the views outside the anchor set at a cached step. */
typedef enum {
    GEOCACHE_UPDATE_DELTA = 0, /* Eq. 1: integrate the anchors' transported change of x0 */
    GEOCACHE_UPDATE_COPY = 1   /* value-copy ablation (Sec. 4.3, Table 3 "delta -> copy"): a covered
                                  token takes the anchors' transported x0 itself */
} geocache_update;

/* One kept (target token, source view) row of G_{u->v} in sparse form: the
 * bilinear footprint's top-left tap and fractions, from which the kept taps'
 * indices and renormalised weights follow exactly as in the tables.
 * 16 bytes. */
typedef struct {
    int32_t token_mask;   /* target token p (bits 0..27) | keep mask << 28 (bit k = tap k kept) */
    int32_t q_tl;         /* source index of the top-left tap (row*W + col; may be -1 or -W-1 off-image) */
    float fx, fy;         /* footprint fractions (K = 4); 0 for K = 1, where q_tl is the single tap */
} geocache_tap_record;

/* Pinhole camera, world -> camera: x_c = R x_w + t (R row-major), +z forward,
 * pixel x right, pixel y down, token (i, j) centred at (i + 0.5, j + 0.5).
 * 64 bytes. */
typedef struct {
    float R[9];
    float t[3];
    float fx, fy, cx, cy;
} geocache_camera;

/* Correspondence operator G_{u->v} of one batch of assets (Sec. 3.2,
 * "Correspondence operator"): for target token p of view v, the K taps of
 * source view u around the projection of X = P_v(p) whose 3-D positions lie
 * within tau of X, with area (bilinear) weights renormalised to sum to one;
 * rows without a kept tap are zero.  K = 4 (bilinear footprint) or K = 1
 * (the token containing the projection).
 * tau = tol_frac * diagonal of the box of the asset's foreground texels
 * (tol_frac = 0.01 in the paper).
 * The struct only records caller-owned device buffers; they must stay valid
 * while calls use the struct. */
typedef struct {
    int B, N, H, W, K;
    float tol_frac;
    const float* pos;               /* device [B,N,H,W,3] f32 world positions of each token */
    const uint8_t* valid;           /* device [B,N,H,W] u8, nonzero = foreground */
    const geocache_camera* cams;    /* device [B,N] */
    float* tau;                     /* device [B] f32, written by geocache_build_corr */
    int32_t* idx;                   /* device [B,N(v),N(u),H,W,K] i32 source token index row*W+col,
                                       -1 = tap not kept; or NULL (tables not built).  A TABLE-mode
                                       step drops an index outside [-1, H*W) and reports it through
                                       the device status word (EINVAL) */
    float* w;                       /* device [B,N(v),N(u),H,W,K] f32 weights, 0 where idx = -1; or NULL */
    uint8_t* keep;                  /* device [B,N(v),N(u),H,W] u8: bit k set iff tap k is kept; or NULL */
    int32_t* tile_ptr;              /* device [B*N*N*T + 1] i32 (T = ceil(H*W / GEOCACHE_TILE_TOKENS)):
                                       records of (b, v, u, tile) are records[tile_ptr[i] .. tile_ptr[i+1]),
                                       i = ((b*N + v)*N + u)*T + tile; or NULL */
    geocache_tap_record* records;   /* device [max_records], sorted by (b, v, u, token); or NULL */
    int64_t max_records;            /* capacity of records */
    geocache_corr_mode mode;        /* taps used by geocache_transport_step */
    int32_t* src_ptr;               /* device [B*N*T + 1] i32 or NULL: source index of the records (with
                                       src_rec; needs records).  Group g = (b*N + u)*T + st holds the records
                                       of source view u of asset b whose first kept tap lies in tile st:
                                       entries [g ? src_ptr[g-1] : 0, src_ptr[g]) of src_rec.  Sparse steps
                                       with C >= 8 whose workspace has no room for the increment plane
                                       then apply the records per source tile (same results). */
    int32_t* src_rec;               /* device [max_records][2] i32, 8-byte aligned, or NULL: entries
                                       (record index, target view v); their order within a group is not
                                       specified */
} geocache_corr;

/* Sampler step parameters (Sec. 3.2, closed-form conversion after Eq. 1).
 * DDIM (eta = 0): 0 < a_t < 1 and 0 < a_prev <= 1 are alpha-bar at this step
 * and at the next one:
 *     eps = (x_t - sqrt(a_t) x0) / sqrt(1 - a_t),
 *     x_next = sqrt(a_prev) x0 + sqrt(1 - a_prev) eps.
 * Flow-matching Euler (x_s = (1 - s) x0 + s eps): sigma > 0, sigma_next >= 0:
 *     u = (x_s - x0) / sigma,  x_next = x_s + (sigma_next - sigma) u.
 * The square roots and reciprocals are formed once in double on the host and
 * rounded to float; the per-element arithmetic is float. */
typedef struct {
    geocache_sampler sampler;
    double a_t, a_prev;
    double sigma, sigma_next;
    geocache_pred pred_kind;
    float* pred_out;   /* device f32, same shape as x_next, or NULL (pred_kind must then be NONE) */
} geocache_recon;

/* Full / cached step policy (Sec. 3.2, drift-bounding schedule). Step 0 is
 * always full (no x0(t-1) exists) except under SINGLE_CACHED. */
typedef enum {
    GEOCACHE_SCHED_EVERY_K = 0,       /* full iff step % k == 0 */
    GEOCACHE_SCHED_HEAD_MID_TAIL = 1, /* first `head` steps, step S/2 if mid != 0, last `tail` steps */
    GEOCACHE_SCHED_LIST = 2,          /* full iff step is in full_steps[0..n_full_steps) */
    GEOCACHE_SCHED_ALL_FULL = 3,      /* every step full (the a = N gate) */
    GEOCACHE_SCHED_SINGLE_CACHED = 4  /* step 0 is a supplied state; every later step is cached */
} geocache_sched_kind;

typedef struct {
    geocache_sched_kind kind;
    int k;
    int head, mid, tail;
    const int32_t* full_steps;        /* host, for GEOCACHE_SCHED_LIST */
    int n_full_steps;
    int contiguous_rotation;          /* 0: strided rotation (default), 1: contiguous blocks */
} geocache_schedule;

/* --------------------------------------------------------------------------
 * geocache_build_corr -- tau and the correspondence tables (Sec. 3.2,
 * "Correspondence operator"; precomputed once per asset).
 *
 * Reads corr->pos, corr->valid, corr->cams; writes corr->tau[B] and, for
 * every ordered pair (v, u), the tables idx/w (when both are non-NULL) and
 * the keep masks (when keep is non-NULL): the diagonal u == v and
 * background targets hold idx -1 / w 0 / keep 0.  When tile_ptr is given
 * (it needs keep) the tile offsets of the sparse form are written, when
 * records is also given the records are written, and when src_ptr and
 * src_rec are also given the source index is written.  The call is asynchronous;
 * size records with geocache_corr_record_count (the count depends only on
 * the geometry).  Records beyond max_records are dropped and flagged in the
 * device status word (geocache_device_status then returns ESHAPE).
 * Sizes: 1 <= B, 2 <= N <= GEOCACHE_MAX_VIEWS, 1 <= H, W <= 16384,
 * K in {1, 4}, 0 < tol_frac.  Outputs must not overlap the inputs.
 * Returns GEOCACHE_OK, EINVAL (NULL / bad K / tol_frac), ESHAPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_build_corr(geocache_corr* corr, void* stream);

/* --------------------------------------------------------------------------
 * geocache_corr_record_count -- number of sparse records of a batch (the
 * kept (target token, source view) rows of every G_{u->v}): builds tau, the
 * keep masks and tile_ptr (corr->keep and corr->tile_ptr are required), then
 * synchronises `stream` and returns the count in *count.  Allocate
 * max_records >= *count records and call geocache_build_corr to fill them.
 * Returns GEOCACHE_OK, EINVAL, ESHAPE, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_corr_record_count(geocache_corr* corr, int64_t* count, void* stream);

/* --------------------------------------------------------------------------
 * geocache_transport_workspace -- number of floats of workspace to give
 * geocache_transport_step for `corr` with C channels: 0 unless corr->mode is
 * GEOCACHE_CORR_SPARSE; then max_records * C (the minimum a step with a < N
 * accepts), plus for C >= 8 room for the anchors' increment plane of any
 * a < N, B * (N-1) * 4*ceil(C/4) * H * W floats.  A step with C >= 8 whose
 * workspace holds max_records * C + B * a * 4*ceil(C/4) * H * W floats
 * writes the plane and gathers the increments from it (faster); with less it
 * applies the records into workspace rows.  Both give the same bits.  Host
 * only.
 * ------------------------------------------------------------------------ */
int64_t geocache_transport_workspace(const geocache_corr* corr, int C);

/* --------------------------------------------------------------------------
 * geocache_transport_step -- one cached sampler step (Eq. 1 and the
 * multi-anchor aggregation, invalid-match and loop-order paragraphs of
 * Sec. 3.2), fused with the sampler reconstruction when recon != NULL.
 *
 *   anchors   host [a], ascending, distinct, in [0, N): the views the
 *             denoiser ran on at this step (1 <= a <= N).
 *   x0_anchor_new  device [B,a,C,H,W] f32: the denoiser's x0 for the anchors,
 *             in the order of `anchors`.
 *   x0_prev   device [B,N,C,H,W] f32: stored x0(t-1) of every view.
 *   x0_out    device [B,N,C,H,W] f32: receives x0(t) of every view:
 *             anchors: x0_anchor_new; other views v:
 *               x0_prev^v + (1/n) sum_{u in A with a kept tap} sum_k w_k Delta^u[q_k],
 *             Delta^u = x0_anchor_new^u - x0_prev^u, n = number of such u;
 *             n = 0 keeps x0_prev^v.
 *             x0_out may equal x0_prev (in-place update; the anchors' rows are
 *             then written by a second kernel after the gathers) but must not
 *             otherwise overlap it.
 *   x_t, x_next  device [B,N,C,H,W] of lat_dtype (F32 or BF16): when recon is
 *             non-NULL, x_next = reconstruction of x_t with x0(t) for every
 *             view (bf16 stores round to nearest even); x_next may equal x_t.
 *             Ignored when recon is NULL.
 *   C         1 <= C <= GEOCACHE_MAX_CHANNELS.
 *   workspace device f32 scratch, 16-byte aligned, of workspace_floats floats:
 *             in sparse mode with a < N at least max_records * C
 *             (geocache_transport_workspace(corr, C) selects the fastest
 *             path); NULL when no scratch is needed.  Its contents are not
 *             preserved between calls, and calls sharing a workspace must not
 *             overlap.
 * corr must have been filled by geocache_build_corr (tau; idx/w in
 * GEOCACHE_CORR_TABLE mode; keep in GEOCACHE_CORR_MASK mode; keep, tile_ptr
 * and records in GEOCACHE_CORR_SPARSE mode).
 * Returns GEOCACHE_OK, EINVAL, ESHAPE, EDTYPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_transport_step(const geocache_corr* corr, const int32_t* anchors, int a, int C,
                            const float* x0_anchor_new, const float* x0_prev, float* x0_out,
                            const void* x_t, void* x_next, geocache_dtype lat_dtype,
                            const geocache_recon* recon, float* workspace, int64_t workspace_floats,
                            void* stream);

/* --------------------------------------------------------------------------
 * geocache_transport_step_update -- geocache_transport_step with the update
 * rule of the views outside the anchor set chosen (the ablations of Sec. 4.3).
 * GEOCACHE_UPDATE_DELTA is geocache_transport_step.  GEOCACHE_UPDATE_COPY
 * overwrites instead of integrating: a token of view v with n >= 1 covering
 * anchors gets
 *     x0_out^v = (1/n) sum_{u in A with a kept tap} sum_k w_k x0_anchor_new^u[q_k]
 * and a token with n = 0 keeps x0_prev^v; anchors and the reconstruction are
 * as in geocache_transport_step.  Same arguments, layouts, ownership and
 * statuses as geocache_transport_step, plus EINVAL for an unknown update.
 * ------------------------------------------------------------------------ */
int geocache_transport_step_update(const geocache_corr* corr, geocache_update update, const int32_t* anchors, int a,
                                   int C, const float* x0_anchor_new, const float* x0_prev, float* x0_out,
                                   const void* x_t, void* x_next, geocache_dtype lat_dtype,
                                   const geocache_recon* recon, float* workspace, int64_t workspace_floats,
                                   void* stream);

/* --------------------------------------------------------------------------
 * geocache_permute_records -- the shuffled-correspondence ablation (Sec. 4.3,
 * Table 3 "corr -> shuffled"): the nonzero rows of each G_{u->v} exchange
 * their taps.  out[r] keeps the target token of corr->records[r] and takes
 * the keep mask, top-left tap and fractions of corr->records[perm[r]], for
 * r in [0, corr->max_records).
 *   corr   a sparse-form corr filled by geocache_build_corr (records,
 *          max_records; its other fields are not read).
 *   perm   device [max_records] i32, a permutation of [0, max_records) that
 *          maps the records of each (b, v, u) pair, tile_ptr[i*T] ..
 *          tile_ptr[(i+1)*T) with i = (b*N + v)*N + u, onto themselves (the
 *          caller's seeded input; other permutations give a correspondence
 *          whose rows belong to other pairs).  An entry outside
 *          [0, max_records) leaves out[r] = records[r] and sets the device
 *          status word (geocache_device_status then returns EINVAL).
 *   out    device [max_records] records, 16-byte aligned, overlapping
 *          neither corr->records nor perm.  A corr whose records are `out`
 *          runs the shuffled transport in GEOCACHE_CORR_SPARSE mode.
 * Asynchronous.  Returns GEOCACHE_OK, EINVAL, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_permute_records(const geocache_corr* corr, const int32_t* perm, geocache_tap_record* out, void* stream);

/* --------------------------------------------------------------------------
 * geocache_raster_posmaps -- the position maps and validity masks of B
 * triangle meshes, each seen by N cameras (the rendered position maps of
 * Sec. 3.1 that the correspondence operator of Sec. 3.2 is built from), by a
 * z-buffer over pixel centres: pixel (i, j) is covered by a face when its
 * centre (i + 0.5, j + 0.5) lies inside or on the face's projection (faces
 * with a vertex at camera z <= 1e-6 or zero projected area are skipped);
 * the nearest such face along the pixel's ray wins (ties to the lower face
 * index) and pos holds the world position of that ray / face-plane
 * intersection.  Decisions and positions are binary32, one rounding per
 * operation in a fixed order, so the maps are reproducible bit for bit.
 *   verts     device [n_verts, 3] f32 world positions of all meshes.
 *   faces     device [n_faces, 3] i32 indices into verts; faces of asset b
 *             are faces[face_off[b] .. face_off[b+1]).  A face with an index
 *             outside [0, n_verts) is skipped and reported in the device
 *             status word (geocache_device_status then returns EINVAL).
 *   face_off  device [B + 1] i64, ascending, face_off[0] = 0,
 *             face_off[B] = n_faces (n_faces < 2^32).
 *   cams      device [B, N] cameras (geocache_camera).
 *   zbuf      device [B, N, H, W] u64 scratch (overwritten).
 *   pos, valid  device [B, N, H, W, 3] f32 / [B, N, H, W] u8 outputs, the
 *             layout of geocache_corr.pos / .valid; uncovered pixels get
 *             position 0 and valid 0.
 * Asynchronous.  Sizes: 1 <= B <= 65535, 1 <= N <= GEOCACHE_MAX_VIEWS,
 * 1 <= H, W <= 16384.  Returns GEOCACHE_OK, EINVAL, ESHAPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_raster_posmaps(const float* verts, int64_t n_verts, const int32_t* faces, int64_t n_faces,
                            const int64_t* face_off, int B, const geocache_camera* cams, int N, int H, int W,
                            uint64_t* zbuf, float* pos, uint8_t* valid, void* stream);

/* --------------------------------------------------------------------------
 * geocache_raster_posmaps_supersampled -- geocache_raster_posmaps rendered at
 * s times the token grid and pooled to it.  A pipeline renders its position
 * maps at image resolution (Sec. 3.1; e.g. 512 x 512 views for 64 x 64
 * latents, s = 8), while the correspondence operator acts on the latent
 * token grid (Sec. 3.2).  The faces are rasterised at (s H) x (s W) with each
 * camera's fx, fy, cx, cy multiplied by s (binary32), under the rules of
 * geocache_raster_posmaps; token (i, j) then covers pixels (i s + sx,
 * j s + sy), 0 <= sx, sy < s.  Its position is the mean of the positions of
 * its valid pixels (summed componentwise in binary32, rows sy ascending and
 * sx ascending within a row, then divided once by their number n) and it is
 * foreground when 2 n >= s * s; background tokens get position 0.  s = 1 is
 * geocache_raster_posmaps.
 *   cams      device [B, N] cameras of the token grid (H x W).
 *   zbuf      device [B, N, s H, s W] u64 scratch (overwritten).
 *   pos, valid  device [B, N, H, W, 3] f32 / [B, N, H, W] u8 token-grid maps.
 * Sizes: as geocache_raster_posmaps, 1 <= s <= 16, s H and s W <= 16384.
 * Asynchronous.  Returns GEOCACHE_OK, EINVAL, ESHAPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_raster_posmaps_supersampled(const float* verts, int64_t n_verts, const int32_t* faces, int64_t n_faces,
                                         const int64_t* face_off, int B, const geocache_camera* cams, int N, int H,
                                         int W, int s, uint64_t* zbuf, float* pos, uint8_t* valid, void* stream);

/* --------------------------------------------------------------------------
 * geocache_pool_posmaps -- token-grid position maps from maps the caller
 * rendered at s times the token resolution (Sec. 3.1 / 3.2, as above; the
 * pooling rule of geocache_raster_posmaps_supersampled).
 *   pos_hi, valid_hi  device [n_maps, s H, s W, 3] f32 / [n_maps, s H, s W] u8
 *                     (valid nonzero = foreground).
 *   pos, valid        device [n_maps, H, W, 3] f32 / [n_maps, H, W] u8.
 * Outputs must not overlap the inputs.  Sizes: n_maps >= 0, 1 <= H, W,
 * 1 <= s <= 16, s H and s W <= 16384.  Asynchronous.  Returns GEOCACHE_OK,
 * EINVAL, ESHAPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_pool_posmaps(const float* pos_hi, const uint8_t* valid_hi, int64_t n_maps, int H, int W, int s, float* pos,
                          uint8_t* valid, void* stream);

/* --------------------------------------------------------------------------
 * geocache_reconstruct -- full-step passthrough (Sec. 3.2: at a full step the
 * denoiser runs on all N views and its x0 is both the new reference and the
 * input of the sampler conversion).
 *
 *   x_t, x_next  device [n] of lat_dtype (may be equal);  x0 device [n] f32;
 *   x0_store     device [n] f32 copy of x0 (the stored reference), or NULL.
 * Returns GEOCACHE_OK, EINVAL, ESHAPE (n < 0), EDTYPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_reconstruct(const void* x_t, const float* x0, void* x_next, geocache_dtype lat_dtype,
                         int64_t n, const geocache_recon* recon, float* x0_store, void* stream);

/* --------------------------------------------------------------------------
 * geocache_pack_anchors / geocache_unpack_anchors -- the batch slicing around
 * the denoiser's anchor-only forward (Sec. 3.2, batch-sliced anchor forward:
 * at a cached step only the anchor rows of the batch run the denoiser, each
 * keeping its own structural indices).
 *
 * A per-view tensor is seen as B x N rows of row_bytes bytes (e.g. latents
 * [B,N,C,H,W], conditioning maps, or per-view index tensors).
 *   pack:   dst [B, a, row] receives src [B, N, row] rows of the anchors, in
 *           the order of `anchors` (host [a], ascending, distinct, in [0, N)).
 *   unpack: dst [B, N, row] receives src [B, a, row] at the anchors' rows; the
 *           other rows of dst are left untouched.
 * Both are device copies of raw bytes (any dtype), asynchronous on `stream`;
 * src and dst must not overlap.  Sizes: 0 <= B <= 65535, 1 <= a <= N <= 64,
 * row_bytes >= 0.  Returns GEOCACHE_OK, EINVAL, ESHAPE, EALIAS, ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_pack_anchors(const void* src, void* dst, int64_t row_bytes, int B, int N, const int32_t* anchors, int a,
                          void* stream);
int geocache_unpack_anchors(const void* src, void* dst, int64_t row_bytes, int B, int N, const int32_t* anchors,
                            int a, void* stream);

/* --------------------------------------------------------------------------
 * geocache_is_full_step -- 1 if `step` (0 <= step < S) is a full step under
 * `sched`, 0 if cached, a negative status on bad arguments. Host only.
 * ------------------------------------------------------------------------ */
int geocache_is_full_step(int step, int S, const geocache_schedule* sched);

/* --------------------------------------------------------------------------
 * geocache_rotate_anchors -- anchor set of `step` (Sec. 3.2, batch-sliced
 * anchor forward: the anchors rotate every step and every view returns to the
 * full context every ceil(N/a) steps).  Host only.
 *
 * With r = number of cached steps before `step` under `sched`:
 *   strided (default): s = ceil(N/a), A = {(r mod s + j s) mod N : j < a};
 *   contiguous:        A = {(r a + j) mod N : j < a};
 * a repeated id is replaced by the smallest id not used by A otherwise.
 * anchors_out (host [a]) receives A in ascending order; *is_full_out (may be
 * NULL) receives 1 if the step is a full step (the anchors are then the ones
 * the next cached step will use) and 0 otherwise.
 * Returns GEOCACHE_OK, EINVAL, ESHAPE.
 * ------------------------------------------------------------------------ */
int geocache_rotate_anchors(int N, int a, int step, int S, const geocache_schedule* sched,
                            int32_t* anchors_out, int* is_full_out);

/* --------------------------------------------------------------------------
 * geocache_device_status -- synchronises `stream`, then reads and clears the
 * device status word.  Failures only the GPU can see set it instead of
 * trapping, so the context stays usable: a sparse-form build whose records
 * exceed max_records (the excess is dropped; transport steps read only the
 * records that exist), a record permutation entry out of range
 * (geocache_permute_records keeps that record), a mesh face with a vertex
 * index out of range (geocache_raster_posmaps skips it), a correspondence
 * table index outside [-1, H*W) in a TABLE-mode step (that tap is dropped),
 * and a bounded wait inside a kernel that ran out (its CTA returns without
 * writing its outputs).
 * Returns GEOCACHE_OK, ESHAPE (record overflow), EINVAL (bad permutation
 * entry, face index or table index), ETIMEOUT (a wait gave up) or ECUDA.
 * ------------------------------------------------------------------------ */
int geocache_device_status(void* stream);

/* --------------------------------------------------------------------------
 * geocache_debug_set_wait -- test hook of the failure handling (the paper has
 * no counterpart; not needed in normal use).  The staged transport kernel
 * (GEOMETRY / TABLE / MASK modes with H*W % 8 == 0 and 16-byte aligned
 * buffers) waits for its shared-memory copies with a time limit instead of
 * spinning forever.
 *   limit_ns         limit of those waits for later calls (0 = the default, 2 s).
 *   drop_first_copy  nonzero: the next call that runs the staged kernel arms
 *                    none of the copies of its first unit (asset 0, view 0,
 *                    first tile, first channel group), so that wait runs out
 *                    for certain; its CTA sets the timeout bit of the device
 *                    status word (geocache_device_status then returns
 *                    GEOCACHE_ETIMEOUT) and returns without writing the
 *                    outputs of its units, and the context stays usable.  The
 *                    request is consumed by that call.
 * Process-wide, not thread safe.  Returns GEOCACHE_OK.
 * ------------------------------------------------------------------------ */
int geocache_debug_set_wait(uint64_t limit_ns, int drop_first_copy);

/* --------------------------------------------------------------------------
 * geocache_transport_step_noalloc -- geocache_transport_step for callers that
 * cannot supply a workspace (the paper has no counterpart; this is a service
 * of the library).  Some callers cannot obtain a device buffer where they run
 * a step: their device memory is owned by another component (a framework's
 * caching allocator, a fixed arena), or they must not allocate once running
 * because cudaMalloc can synchronise the device and stall.  This entry point
 * takes the same arguments minus the workspace and allocates nothing: its
 * scratch is a fixed array of GEOCACHE_NOALLOC_MAX_WORKSPACE_FLOATS floats
 * (16 MiB) in the library's device image, present on every device that loads
 * the library until the process exits.
 *  - A step that needs more scratch (a sparse-mode step with a < N whose
 *    max_records * C exceeds the array) is rejected with GEOCACHE_ESHAPE;
 *    steps that need none (a == N, other modes) are always accepted.  The
 *    whole array is passed as the workspace, so a step with C >= 8 takes
 *    the increment-plane path when the array also holds the plane.
 *  - The first call on each device looks up the array's device address with
 *    that device current; make that first call before any stream capture.
 *    The address is kept for the life of the process, so the entry point
 *    must not be used on a device after cudaDeviceReset (or any other
 *    teardown of its primary context) in the same process.
 *  - Every call on a device shares the one array, which keeps the previous
 *    call's contents; nothing in it needs to start at zero (each entry a call
 *    reads is written earlier in the same call), but calls that overlap on
 *    the GPU (e.g. on different streams) race and must not be issued.
 * Returns the statuses of geocache_transport_step.
 * ------------------------------------------------------------------------ */
#define GEOCACHE_NOALLOC_MAX_WORKSPACE_FLOATS (4 * 1024 * 1024)
int geocache_transport_step_noalloc(const geocache_corr* corr, const int32_t* anchors, int a, int C,
                                    const float* x0_anchor_new, const float* x0_prev, float* x0_out,
                                    const void* x_t, void* x_next, geocache_dtype lat_dtype,
                                    const geocache_recon* recon, void* stream);

/* Thread-local description of the last non-OK status of this thread ("" if
 * none).  The pointer stays valid until the thread's next library call. */
const char* geocache_last_error(void);

/* GEOCACHE_ABI_VERSION of the loaded library. */
int geocache_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* GEOCACHE_H */
