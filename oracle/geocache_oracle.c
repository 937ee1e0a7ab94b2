/*
 * GeoCache CPU ORACLE -- test infrastructure, not product code.
 *
 * A plain, slow, single-threaded restatement of the geometric delta transport
 * (Sec. 3.2 of the paper).  Only the tests, the smoke check and the CPU
 * baseline of the benchmark call it.  It shares no code with the CUDA path.
 *
 * Precision:
 *   - Quantities that decide an integer (the tolerance tau, the projection of
 *     a target point into a source camera, the choice of taps and the
 *     position-agreement test) are evaluated in IEEE binary32, one rounding
 *     per operation in the order written below (compile with
 *     -ffp-contract=off so that no multiply-add is fused).
 *   - Everything continuous (tap weights, the transported increment, the
 *     sampler reconstruction) is evaluated in binary64.
 *
 * Camera record (16 floats): R[9] row-major world->camera, t[3], fx, fy, cx,
 * cy; +z forward, pixel y down, pixel (i, j) centred at (i + 0.5, j + 0.5).
 *
 * Readings taken where the paper is silent (each is listed with its reason
 * in the design notes of the repository):
 *   - "K nearest source taps ... area-weight them" (Sec. 3.2, correspondence
 *     operator): the K = 4 pixel centres of the bilinear footprint around the
 *     projection of the target point, weighted by the bilinear (area)
 *     weights; K = 1 is the pixel containing the projection.
 *   - A tap is kept iff it lies in the image, its texel is foreground, its
 *     raw weight is non-zero and its squared 3-D distance to the target point
 *     is <= tau^2 (the per-tap tolerance); kept weights are renormalised to
 *     sum to one, so each row of G_{u->v} sums to one or is zero.
 *   - tau = tol_frac * (diagonal of the axis-aligned box of all foreground
 *     position-map texels of the asset), tol_frac = 0.01.
 *   - Multi-anchor "normalized sum" (Sec. 3.2, multi-anchor aggregation): the
 *     mean of the per-anchor transports over the anchors that have at least
 *     one kept tap.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_MAX_K 4

/* ------------------------------------------------------------------ tau -- */
/* tau per asset (correspondence-operator paragraph, "1% of the bounding-box
 * diagonal").  pos [B,N,H,W,3] f32, valid [B,N,H,W] u8, tau_out [B] f32. */
int oracle_tau(const float* pos, const uint8_t* valid, int B, int N, int H, int W,
               float tol_frac, float* tau_out) {
    if (!pos || !valid || !tau_out || B < 0 || N <= 0 || H <= 0 || W <= 0) return -1;
    const size_t per_asset = (size_t)N * H * W;
    for (int b = 0; b < B; ++b) {
        float lo[3] = {INFINITY, INFINITY, INFINITY};
        float hi[3] = {-INFINITY, -INFINITY, -INFINITY};
        int any = 0;
        for (size_t i = 0; i < per_asset; ++i) {
            const size_t g = (size_t)b * per_asset + i;
            if (!valid[g]) continue;
            any = 1;
            for (int c = 0; c < 3; ++c) {
                const float x = pos[3 * g + c];
                if (x < lo[c]) lo[c] = x;
                if (x > hi[c]) hi[c] = x;
            }
        }
        if (!any) { tau_out[b] = 0.0f; continue; }
        const float d0 = hi[0] - lo[0], d1 = hi[1] - lo[1], d2 = hi[2] - lo[2];
        const float diag2 = (d0 * d0 + d1 * d1) + d2 * d2;
        tau_out[b] = tol_frac * sqrtf(diag2);
    }
    return 0;
}

/* ----------------------------------------------------------- projection -- */
/* x_c = R X + t, then the pinhole projection; returns 0 when the point is not
 * in front of the camera. */
int oracle_project(const float* cam, const float* X, float* uu, float* vv) {
    float xc[3];
    for (int r = 0; r < 3; ++r) {
        float s = cam[3 * r] * X[0];
        s = s + cam[3 * r + 1] * X[1];
        s = s + cam[3 * r + 2] * X[2];
        xc[r] = s + cam[9 + r];
    }
    if (!(xc[2] > 0.0f)) return 0;
    const float qx = xc[0] / xc[2];
    const float qy = xc[1] / xc[2];
    *uu = cam[12] * qx + cam[14];
    *vv = cam[13] * qy + cam[15];
    return 1;
}

static float sqdist(const float* a, const float* b) {
    const float dx = a[0] - b[0], dy = a[1] - b[1], dz = a[2] - b[2];
    return (dx * dx + dy * dy) + dz * dz;
}

/* Taps of one target point X (a foreground texel of view v) in source view u.
 * pos_u [H,W,3], valid_u [H,W].  Writes K linear source indices (row*W+col,
 * -1 when the tap is not kept) and K binary64 weights (0 when not kept).
 * Returns the number of kept taps.  *band is set when some tap that passed
 * every test but the distance test, or passed it, has a binary64 distance
 * within 1e-6 of tau (the threshold band counted by the tests). */
int oracle_taps(const float* cam_u, const float* pos_u, const uint8_t* valid_u, int H, int W,
                const float* X, float tau, int K, int32_t* idx, double* w, int* band) {
    for (int k = 0; k < K; ++k) { idx[k] = -1; w[k] = 0.0; }
    if (band) *band = 0;
    float uu, vv;
    if (!oracle_project(cam_u, X, &uu, &vv)) return 0;
    const float tau2 = tau * tau;
    int cols[ORC_MAX_K], rows[ORC_MAX_K];
    double raw[ORC_MAX_K];
    int nz[ORC_MAX_K];
    if (K == 1) {
        if (!(uu >= 0.0f && uu < (float)W && vv >= 0.0f && vv < (float)H)) return 0;
        cols[0] = (int)floorf(uu);
        rows[0] = (int)floorf(vv);
        raw[0] = 1.0;
        nz[0] = 1;
    } else if (K == 4) {
        const float x = uu - 0.5f, y = vv - 0.5f;
        if (!(x >= -1.0f && x < (float)W && y >= -1.0f && y < (float)H)) return 0;
        const float i0f = floorf(x), j0f = floorf(y);
        const int i0 = (int)i0f, j0 = (int)j0f;
        const float fx = x - i0f, fy = y - j0f;
        const float ax[2] = {1.0f - fx, fx};
        const float ay[2] = {1.0f - fy, fy};
        for (int k = 0; k < 4; ++k) {
            const int di = k & 1, dj = k >> 1;
            cols[k] = i0 + di;
            rows[k] = j0 + dj;
            nz[k] = (ax[di] != 0.0f) && (ay[dj] != 0.0f);
            raw[k] = (double)ax[di] * (double)ay[dj]; /* exact in binary64 */
        }
    } else {
        return 0;
    }
    double sum = 0.0;
    int kept = 0;
    for (int k = 0; k < K; ++k) {
        if (cols[k] < 0 || cols[k] >= W || rows[k] < 0 || rows[k] >= H) continue;
        const int q = rows[k] * W + cols[k];
        if (!valid_u[q] || !nz[k]) continue;
        const float* Pq = pos_u + 3 * (size_t)q;
        if (band) {
            const double dx = (double)Pq[0] - X[0], dy = (double)Pq[1] - X[1], dz = (double)Pq[2] - X[2];
            if (fabs(sqrt(dx * dx + dy * dy + dz * dz) - (double)tau) <= 1e-6) *band = 1;
        }
        if (!(sqdist(Pq, X) <= tau2)) continue;
        idx[k] = q;
        sum += raw[k];
        ++kept;
    }
    for (int k = 0; k < K; ++k)
        if (idx[k] >= 0) w[k] = raw[k] / sum;
    return kept;
}

/* -------------------------------------------------- correspondence build -- */
/* Tables of G_{u->v} for every ordered pair: idx/w [B, N(target v), N(source
 * u), H, W, K]; the diagonal u == v and background targets hold -1 / 0.
 * band_out [B,N,N,H,W] (optional) flags target pixels in the threshold band.
 * Returns the number of flagged pixels (>= 0) or -1 on bad arguments. */
long oracle_build_corr(const float* pos, const uint8_t* valid, const float* cams, const float* tau,
                       int B, int N, int H, int W, int K, int32_t* idx, double* w, uint8_t* band_out) {
    if (!pos || !valid || !cams || !tau || !idx || !w || (K != 1 && K != 4)) return -1;
    const size_t HW = (size_t)H * W;
    long nband = 0;
    for (int b = 0; b < B; ++b)
        for (int v = 0; v < N; ++v)
            for (int u = 0; u < N; ++u)
                for (size_t p = 0; p < HW; ++p) {
                    const size_t row = (((size_t)b * N + v) * N + u) * HW + p;
                    int32_t* ri = idx + row * K;
                    double* rw = w + row * K;
                    int bd = 0;
                    const size_t tv = ((size_t)b * N + v) * HW + p;
                    if (u == v || !valid[tv]) {
                        for (int k = 0; k < K; ++k) { ri[k] = -1; rw[k] = 0.0; }
                    } else {
                        const size_t su = ((size_t)b * N + u) * HW;
                        oracle_taps(cams + ((size_t)b * N + u) * 16, pos + 3 * su, valid + su, H, W,
                                    pos + 3 * tv, tau[b], K, ri, rw, &bd);
                    }
                    if (band_out) band_out[row] = (uint8_t)bd;
                    nband += bd;
                }
    return nband;
}

/* Brute-force restatement of one row of G_{u->v} used to pin the tap logic:
 * every source texel q gets the tent weight
 *   max(0, 1-|q_x+0.5-uu|) * max(0, 1-|q_y+0.5-vv|)        (K = 4)
 * or the indicator that (uu, vv) lies in q's pixel square  (K = 1),
 * masked by foreground and by the binary64 tolerance test, then normalised.
 * There is no floor and no tap list.  Writes at most 4 (index, weight) pairs
 * in ascending index order; returns their count. */
int oracle_brute_row(const float* cam_u, const float* pos_u, const uint8_t* valid_u, int H, int W,
                     const float* X, float tau, int K, int32_t* q_out, double* w_out) {
    float uu, vv;
    int n = 0;
    if (!oracle_project(cam_u, X, &uu, &vv)) return 0;
    double sum = 0.0;
    const double t2 = (double)tau * (double)tau;
    for (int r = 0; r < H; ++r)
        for (int c = 0; c < W; ++c) {
            double wt;
            if (K == 4) {
                const double ex = 1.0 - fabs((double)c + 0.5 - (double)uu);
                const double ey = 1.0 - fabs((double)r + 0.5 - (double)vv);
                wt = (ex > 0.0 ? ex : 0.0) * (ey > 0.0 ? ey : 0.0);
            } else {
                wt = ((double)uu >= c && (double)uu < c + 1.0 && (double)vv >= r && (double)vv < r + 1.0) ? 1.0 : 0.0;
            }
            if (wt <= 0.0) continue;
            const int q = r * W + c;
            if (!valid_u[q]) continue;
            const float* Pq = pos_u + 3 * (size_t)q;
            const double dx = (double)Pq[0] - X[0], dy = (double)Pq[1] - X[1], dz = (double)Pq[2] - X[2];
            if (!(dx * dx + dy * dy + dz * dz <= t2)) continue;
            if (n >= 4) return -1;
            q_out[n] = q;
            w_out[n] = wt;
            sum += wt;
            ++n;
        }
    for (int i = 0; i < n; ++i) w_out[i] /= sum;
    return n;
}

/* ------------------------------------------------------ reconstruction -- */
enum { ORC_DDIM = 0, ORC_FM_EULER = 1 };
enum { ORC_PRED_NONE = 0, ORC_PRED_EPS = 1, ORC_PRED_V = 2, ORC_PRED_VELOCITY = 3 };

typedef struct {
    int sampler;      /* ORC_DDIM / ORC_FM_EULER */
    double a_t, a_prev;          /* DDIM: alpha-bar at this step and the next */
    double sigma, sigma_next;    /* flow matching */
    int pred_kind;
} orc_recon;

/* Sampler-consistent reconstruction of one element (Sec. 3.2, last paragraph
 * before Table 1): from x_t and the (transported) x0 compute the sampler's
 * native quantity and take the step.
 *   DDIM (eta = 0): eps = (x_t - sqrt(ab_t) x0) / sqrt(1 - ab_t),
 *                   x_prev = sqrt(ab_prev) x0 + sqrt(1 - ab_prev) eps,
 *                   v = sqrt(ab_t) eps - sqrt(1 - ab_t) x0.
 *   Flow-matching Euler (x_s = (1 - s) x0 + s eps): velocity u = (x_s - x0)/s,
 *                   x_{s'} = x_s + (s' - s) u. */
static void recon_one(const orc_recon* r, double xt, double x0, double* x_next, double* pred) {
    if (r->sampler == ORC_DDIM) {
        const double st = sqrt(r->a_t), s1t = sqrt(1.0 - r->a_t);
        const double sp = sqrt(r->a_prev), s1p = sqrt(1.0 - r->a_prev);
        const double eps = (xt - st * x0) / s1t;
        *x_next = sp * x0 + s1p * eps;
        if (pred) *pred = (r->pred_kind == ORC_PRED_V) ? st * eps - s1t * x0 : eps;
    } else {
        const double vel = (xt - x0) / r->sigma;
        *x_next = xt + (r->sigma_next - r->sigma) * vel;
        if (pred) *pred = vel;
    }
}

int oracle_reconstruct(const double* x_t, const double* x0, double* x_next, double* pred, long n,
                       int sampler, double a_t, double a_prev, double sigma, double sigma_next,
                       int pred_kind) {
    const orc_recon r = {sampler, a_t, a_prev, sigma, sigma_next, pred_kind};
    if (sampler == ORC_DDIM && !(a_t < 1.0)) return -1;
    if (sampler == ORC_FM_EULER && !(sigma > 0.0)) return -1;
    for (long i = 0; i < n; ++i)
        recon_one(&r, x_t[i], x0[i], &x_next[i], (pred && pred_kind) ? &pred[i] : NULL);
    return 0;
}

/* ----------------------------------------------------- delta transport -- */
/* One cached step (Eq. 1 with the multi-anchor aggregation, the invalid-match
 * rule and the loop order of Sec. 3.2):
 *   anchors u in A:   x0^u(t) = x0_new^u  (the denoiser's output),
 *   other views v:    x0^v(t) = x0^v(t-1) + (1/n) sum_{u in A covering p}
 *                               sum_k w_k(p) (x0_new^u - x0^u(t-1))[q_k],
 *                     n = number of anchors with a kept tap; n = 0 keeps
 *                     x0^v(t-1) unchanged,
 * then (optionally) the reconstruction of x_{t-1} for every view.
 * Taps come from a table (idx/w [B,N,N,H,W,K], when idx != NULL) or are
 * computed from the geometry (pos/valid/cams/tau) with oracle_taps.
 * Layouts: x0_new [B,a,C,H,W]; x0_prev, x0_out, x_t, x_next, pred [B,N,C,H,W].
 * Only target pixels with sel[b*N*HW + v*HW + p] != 0 are written when sel
 * is given (sampled checks at large sizes).
 * copy != 0 is the value-copy ablation of Sec. 4.3 ("delta -> copy"): a
 * covered target takes the anchors' transported x0 itself,
 *     x0^v(t) = (1/n) sum_{u in A covering p} sum_k w_k(p) x0_new^u[q_k],
 * and an uncovered one keeps x0^v(t-1). */
int oracle_transport_step(int B, int N, int H, int W, int K, int C,
                          const int32_t* idx, const double* wtab,
                          const float* pos, const uint8_t* valid, const float* cams, const float* tau,
                          const int* anchors, int a,
                          const double* x0_new, const double* x0_prev, double* x0_out,
                          const double* x_t, double* x_next, double* pred,
                          int sampler, double a_t, double a_prev, double sigma, double sigma_next,
                          int pred_kind, const uint8_t* sel, int copy) {
    if (a < 1 || a > N || C < 1 || (K != 1 && K != 4)) return -1;
    if (!idx && (!pos || !valid || !cams || !tau)) return -1;
    int slot_of[256];
    if (N > 256) return -1;
    for (int v = 0; v < N; ++v) slot_of[v] = -1;
    for (int s = 0; s < a; ++s) {
        if (anchors[s] < 0 || anchors[s] >= N || slot_of[anchors[s]] >= 0) return -1;
        if (s > 0 && anchors[s] <= anchors[s - 1]) return -1;
        slot_of[anchors[s]] = s;
    }
    const orc_recon r = {sampler, a_t, a_prev, sigma, sigma_next, pred_kind};
    const size_t HW = (size_t)H * W;
    double* acc = (double*)malloc(sizeof(double) * (size_t)C);
    if (!acc) return -2;
    for (int b = 0; b < B; ++b)
        for (int v = 0; v < N; ++v)
            for (size_t p = 0; p < HW; ++p) {
                if (sel && !sel[((size_t)b * N + v) * HW + p]) continue;
                const size_t plane0 = ((size_t)b * N + v) * C * HW + p; /* element (b,v,0,p) */
                if (slot_of[v] >= 0) {
                    const size_t nw = ((size_t)b * a + slot_of[v]) * C * HW + p;
                    for (int c = 0; c < C; ++c) x0_out[plane0 + c * HW] = x0_new[nw + c * HW];
                } else {
                    int n = 0;
                    for (int c = 0; c < C; ++c) acc[c] = 0.0;
                    for (int s = 0; s < a; ++s) {
                        const int u = anchors[s];
                        int32_t ti[ORC_MAX_K];
                        double tw[ORC_MAX_K];
                        int kept = 0;
                        if (idx) {
                            const size_t row = (((size_t)b * N + v) * N + u) * HW + p;
                            for (int k = 0; k < K; ++k) {
                                ti[k] = idx[row * K + k];
                                tw[k] = wtab[row * K + k];
                                kept += ti[k] >= 0;
                            }
                        } else {
                            const size_t tv = ((size_t)b * N + v) * HW + p;
                            const size_t su = ((size_t)b * N + u) * HW;
                            if (valid[tv])
                                kept = oracle_taps(cams + ((size_t)b * N + u) * 16, pos + 3 * su, valid + su,
                                                   H, W, pos + 3 * tv, tau[b], K, ti, tw, NULL);
                        }
                        if (!kept) continue;
                        ++n;
                        const size_t nw = ((size_t)b * a + s) * C * HW;
                        const size_t pu = ((size_t)b * N + u) * C * HW;
                        for (int c = 0; c < C; ++c) {
                            double g = 0.0;
                            for (int k = 0; k < K; ++k) {
                                if (ti[k] < 0) continue;
                                const size_t q = (size_t)c * HW + (size_t)ti[k];
                                /* Eq. 1 carries the anchor's change; the value-copy
                                   ablation (Sec. 4.3) carries its x0 itself */
                                g += tw[k] * (copy ? x0_new[nw + q] : x0_new[nw + q] - x0_prev[pu + q]);
                            }
                            acc[c] += g;
                        }
                    }
                    for (int c = 0; c < C; ++c)
                        x0_out[plane0 + c * HW] = !n    ? x0_prev[plane0 + c * HW]
                                                  : copy ? acc[c] / n
                                                         : x0_prev[plane0 + c * HW] + acc[c] / n;
                }
                if (x_t && x_next)
                    for (int c = 0; c < C; ++c) {
                        const size_t e = plane0 + c * HW;
                        recon_one(&r, x_t[e], x0_out[e], &x_next[e], (pred && pred_kind) ? &pred[e] : NULL);
                    }
            }
    free(acc);
    return 0;
}

/* ---------------------------------------------------------------- bf16 -- */
/* Round binary64 to bfloat16 (1 sign, 8 exponent, 7 fraction bits) to nearest,
 * ties to even, straight from the definition: scale the significand to 8
 * bits, round, renormalise.  Handles zero, subnormal results, overflow to
 * infinity and NaN. */
static uint16_t bf16_from_double(double x) {
    if (isnan(x)) return 0x7FC0;
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double m = fabs(x);
    if (m == 0.0) return sign;
    if (isinf(m)) return sign | 0x7F80;
    int e;
    double f = frexp(m, &e); /* m = f * 2^e, f in [0.5, 1) */
    /* normal bf16 numbers have unbiased exponent E = e - 1 in [-126, 127] */
    int E = e - 1;
    int shift = 8; /* significand bits kept (including the implicit one) */
    if (E < -126) shift = 8 - (-126 - E); /* subnormal: fewer bits */
    double scaled = ldexp(f, shift);   /* in [2^(shift-1), 2^shift) */
    double fl = floor(scaled);
    double rem = scaled - fl;
    double q = fl;
    if (rem > 0.5 || (rem == 0.5 && fmod(fl, 2.0) != 0.0)) q = fl + 1.0;
    double val = ldexp(q, e - shift); /* rounded magnitude */
    if (val == 0.0) return sign;
    int e2;
    double f2 = frexp(val, &e2);
    int E2 = e2 - 1;
    if (E2 > 127) return sign | 0x7F80;
    if (E2 < -126) { /* subnormal: value = frac * 2^-133 */
        uint16_t frac = (uint16_t)ldexp(val, 133);
        return sign | frac;
    }
    uint16_t frac = (uint16_t)(ldexp(f2, 8) - 128.0); /* 7 fraction bits */
    return sign | (uint16_t)((E2 + 127) << 7) | frac;
}

void oracle_round_bf16(const double* x, uint16_t* out, long n) {
    for (long i = 0; i < n; ++i) out[i] = bf16_from_double(x[i]);
}

/* ------------------------------------------------------ position maps -- */
/* The rendered position map of one mesh seen by one camera (Sec. 3.1: the
 * per-pixel 3-D coordinates a geometry-conditioned texturing pipeline renders
 * for each view, from which the correspondence operator of Sec. 3.2 is
 * built).  A plain face-major z-buffer:
 *   - a face is skipped when a vertex is not in front (camera z <= 1e-6) or
 *     its projected signed area is 0;
 *   - pixel (i, j) is covered when its centre (i + 0.5, j + 0.5) lies inside
 *     or on the projected triangle: the three edge functions, each zero on
 *     one edge, all have the sign of the area;
 *   - its depth is the camera z of the intersection of the ray through the
 *     centre with the face's plane, which must be positive;
 *   - the nearest face wins, ties going to the lower face index;
 *   - the stored position is that intersection in world coordinates.
 * Every step is binary32, one rounding per operation in the order written
 * (the decisions are the rasteriser's own; the position is exact to those
 * roundings).  V [nv,3] world, F [nf,3] vertex indices, cam 16 floats;
 * pos_out [H,W,3], valid_out [H,W].  Faces with an index outside [0, nv)
 * are skipped.  Returns 0, or -1 on bad arguments, -2 on allocation failure. */
typedef struct {
    float R[9], t[3], fx, fy, cx, cy;
} orc_cam32;

static void raster_cam_point(const orc_cam32* c, const float* X, float* xc) {
    for (int r = 0; r < 3; ++r) {
        float s = c->R[3 * r] * X[0];
        s = s + c->R[3 * r + 1] * X[1];
        s = s + c->R[3 * r + 2] * X[2];
        xc[r] = s + c->t[r];
    }
}

/* depth of the ray through (pu, pv) on the plane (n, nd); 0 when there is none */
static float raster_depth(const orc_cam32* c, const float* n, float nd, float pu, float pv, float* d) {
    d[0] = (pu - c->cx) / c->fx;
    d[1] = (pv - c->cy) / c->fy;
    d[2] = 1.0f;
    float den = n[0] * d[0];
    den = den + n[1] * d[1];
    den = den + n[2];
    if (den == 0.0f) return 0.0f;
    const float s = nd / den;
    return (s > 0.0f && s <= 3.0e38f) ? s : 0.0f;
}

int oracle_raster(const float* V, int nv, const int32_t* F, int nf, const float* cam, int H, int W,
                  float* pos_out, uint8_t* valid_out) {
    if (!V || !F || !cam || !pos_out || !valid_out || nv < 0 || nf < 0 || H <= 0 || W <= 0) return -1;
    orc_cam32 c;
    for (int i = 0; i < 9; ++i) c.R[i] = cam[i];
    for (int i = 0; i < 3; ++i) c.t[i] = cam[9 + i];
    c.fx = cam[12]; c.fy = cam[13]; c.cx = cam[14]; c.cy = cam[15];
    const size_t HW = (size_t)H * W;
    float* depth = (float*)malloc(sizeof(float) * HW);
    int32_t* owner = (int32_t*)malloc(sizeof(int32_t) * HW);
    if (!depth || !owner) { free(depth); free(owner); return -2; }
    for (size_t p = 0; p < HW; ++p) { depth[p] = INFINITY; owner[p] = -1; }
    for (int f = 0; f < nf; ++f) {
        float P[3][3], u[3], v[3];
        int ok = 1;
        for (int k = 0; k < 3; ++k) {
            const int32_t vi = F[3 * (size_t)f + k];
            if (vi < 0 || vi >= nv) { ok = 0; break; }
            raster_cam_point(&c, V + 3 * (size_t)vi, P[k]);
            if (!(P[k][2] > 1e-6f)) { ok = 0; break; }
            u[k] = c.fx * (P[k][0] / P[k][2]) + c.cx;
            v[k] = c.fy * (P[k][1] / P[k][2]) + c.cy;
        }
        if (!ok) continue;
        const float area = (u[1] - u[0]) * (v[2] - v[0]) - (v[1] - v[0]) * (u[2] - u[0]);
        if (!(area > 0.0f || area < 0.0f)) continue;
        const float umin = fminf(u[0], fminf(u[1], u[2])), umax = fmaxf(u[0], fmaxf(u[1], u[2]));
        const float vmin = fminf(v[0], fminf(v[1], v[2])), vmax = fmaxf(v[0], fmaxf(v[1], v[2]));
        const float ilo = fmaxf(ceilf(umin - 0.5f), 0.0f), ihi = fminf(floorf(umax - 0.5f), (float)(W - 1));
        const float jlo = fmaxf(ceilf(vmin - 0.5f), 0.0f), jhi = fminf(floorf(vmax - 0.5f), (float)(H - 1));
        if (!(ilo <= ihi && jlo <= jhi)) continue;
        float e1[3], e2[3], n[3];
        for (int r = 0; r < 3; ++r) { e1[r] = P[1][r] - P[0][r]; e2[r] = P[2][r] - P[0][r]; }
        n[0] = e1[1] * e2[2] - e1[2] * e2[1];
        n[1] = e1[2] * e2[0] - e1[0] * e2[2];
        n[2] = e1[0] * e2[1] - e1[1] * e2[0];
        float nd = n[0] * P[0][0];
        nd = nd + n[1] * P[0][1];
        nd = nd + n[2] * P[0][2];
        for (int j = (int)jlo; j <= (int)jhi; ++j) {
            const float pv = (float)j + 0.5f;
            for (int i = (int)ilo; i <= (int)ihi; ++i) {
                const float pu = (float)i + 0.5f;
                const float w0 = (u[2] - u[1]) * (pv - v[1]) - (v[2] - v[1]) * (pu - u[1]);
                const float w1 = (u[0] - u[2]) * (pv - v[2]) - (v[0] - v[2]) * (pu - u[2]);
                const float w2 = (u[1] - u[0]) * (pv - v[0]) - (v[1] - v[0]) * (pu - u[0]);
                const int in = area > 0.0f ? (w0 >= 0.0f && w1 >= 0.0f && w2 >= 0.0f)
                                           : (w0 <= 0.0f && w1 <= 0.0f && w2 <= 0.0f);
                if (!in) continue;
                float d[3];
                const float s = raster_depth(&c, n, nd, pu, pv, d);
                if (s == 0.0f) continue;
                const size_t p = (size_t)j * W + i;
                if (s < depth[p] || (s == depth[p] && f < owner[p])) { depth[p] = s; owner[p] = f; }
            }
        }
    }
    for (size_t p = 0; p < HW; ++p) {
        float* X = pos_out + 3 * p;
        X[0] = X[1] = X[2] = 0.0f;
        valid_out[p] = owner[p] >= 0;
        if (owner[p] < 0) continue;
        /* the winner's plane and ray again, then world = R^T (x_c - t) */
        const int f = owner[p];
        float P[3][3], e1[3], e2[3], n[3], d[3];
        for (int k = 0; k < 3; ++k) raster_cam_point(&c, V + 3 * (size_t)F[3 * (size_t)f + k], P[k]);
        for (int r = 0; r < 3; ++r) { e1[r] = P[1][r] - P[0][r]; e2[r] = P[2][r] - P[0][r]; }
        n[0] = e1[1] * e2[2] - e1[2] * e2[1];
        n[1] = e1[2] * e2[0] - e1[0] * e2[2];
        n[2] = e1[0] * e2[1] - e1[1] * e2[0];
        float nd = n[0] * P[0][0];
        nd = nd + n[1] * P[0][1];
        nd = nd + n[2] * P[0][2];
        const float s = raster_depth(&c, n, nd, (float)(p % W) + 0.5f, (float)(p / W) + 0.5f, d);
        const float xc[3] = {s * d[0] - c.t[0], s * d[1] - c.t[1], s - c.t[2]};
        for (int r = 0; r < 3; ++r) {
            float x = c.R[r] * xc[0];
            x = x + c.R[3 + r] * xc[1];
            X[r] = x + c.R[6 + r] * xc[2];
        }
    }
    free(depth);
    free(owner);
    return 0;
}

/* ---------------------------------------------------------------- pooling --
 * Position maps rendered at image resolution brought to the latent token
 * grid (Sec. 3.1: the pipeline renders its position maps at image
 * resolution, an s-fold super-sampling of the token grid; Sec. 3.2: the
 * correspondence operator acts on the token grid).  Token (i, j) covers the
 * s x s image pixels (i s + sx, j s + sy), 0 <= sx, sy < s.  Its position is
 * the mean of the positions of its valid pixels: summed componentwise in
 * binary32, pixel rows sy ascending and within a row sx ascending, then
 * divided once by their number n (binary32, correctly rounded).  It is
 * foreground when at least half of its s*s pixels are valid (2 n >= s*s);
 * background tokens get position 0.
 * pos_hi [H*s, W*s, 3], valid_hi [H*s, W*s] -> pos [H, W, 3], valid [H, W].
 * Returns 0, or -1 on bad arguments. */
int oracle_pool(const float* pos_hi, const uint8_t* valid_hi, int H, int W, int s, float* pos, uint8_t* valid) {
    if (!pos_hi || !valid_hi || !pos || !valid || H <= 0 || W <= 0 || s <= 0) return -1;
    const size_t Ws = (size_t)W * s;
    for (int j = 0; j < H; ++j)
        for (int i = 0; i < W; ++i) {
            float sum[3] = {0.0f, 0.0f, 0.0f};
            int n = 0;
            for (int sy = 0; sy < s; ++sy)
                for (int sx = 0; sx < s; ++sx) {
                    const size_t q = ((size_t)j * s + sy) * Ws + (size_t)i * s + sx;
                    if (!valid_hi[q]) continue;
                    for (int c = 0; c < 3; ++c) sum[c] = sum[c] + pos_hi[3 * q + c];
                    ++n;
                }
            const size_t p = (size_t)j * W + i;
            const int fg = 2 * n >= s * s && n > 0;
            valid[p] = (uint8_t)fg;
            for (int c = 0; c < 3; ++c) pos[3 * p + c] = fg ? sum[c] / (float)n : 0.0f;
        }
    return 0;
}
