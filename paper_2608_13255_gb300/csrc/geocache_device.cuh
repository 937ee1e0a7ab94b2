// Device-side geometry of the correspondence operator G_{u->v} (Sec. 3.2,
// "Correspondence operator"): projection of a target token's 3-D position
// into a source camera, choice of the K taps, the per-tap tolerance test and
// the renormalised area weights.
//
// The same functions serve the table build and the on-the-fly taps of the
// transport kernel, so both produce identical indices and weights.  Every
// operation that feeds an integer decision (projection, floor, tolerance
// test) is an explicitly rounded binary32 intrinsic in a fixed order, so no
// multiply-add is ever contracted and the decisions do not depend on how the
// compiler schedules the code.
#pragma once

#include <cstdint>

#include "geocache.h"

namespace geocache {

struct Taps {
    int32_t q[4];   // source token index row*W + col, -1 = not kept
    float w[4];     // renormalised weight, 0 where not kept
    int kept;       // number of kept taps
};

__device__ __forceinline__ void taps_clear(Taps& t) {
#pragma unroll
    for (int k = 0; k < 4; ++k) { t.q[k] = -1; t.w[k] = 0.0f; }
    t.kept = 0;
}

// x_c = R X + t with each row summed ((R0 X0 + R1 X1) + R2 X2) + t, then the
// pinhole projection.  Returns false when the point is not in front.
__device__ __forceinline__ bool project(const geocache_camera& c, float X0, float X1, float X2,
                                        float& uu, float& vv) {
    float xc[3];
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        float s = __fmul_rn(c.R[3 * r], X0);
        s = __fadd_rn(s, __fmul_rn(c.R[3 * r + 1], X1));
        s = __fadd_rn(s, __fmul_rn(c.R[3 * r + 2], X2));
        xc[r] = __fadd_rn(s, c.t[r]);
    }
    if (!(xc[2] > 0.0f)) return false;
    uu = __fadd_rn(__fmul_rn(c.fx, __fdiv_rn(xc[0], xc[2])), c.cx);
    vv = __fadd_rn(__fmul_rn(c.fy, __fdiv_rn(xc[1], xc[2])), c.cy);
    return true;
}

__device__ __forceinline__ float sqdist(const float* P, float X0, float X1, float X2) {
    const float dx = __fsub_rn(__ldg(P + 0), X0);
    const float dy = __fsub_rn(__ldg(P + 1), X1);
    const float dz = __fsub_rn(__ldg(P + 2), X2);
    return __fadd_rn(__fadd_rn(__fmul_rn(dx, dx), __fmul_rn(dy, dy)), __fmul_rn(dz, dz));
}

// Footprint of target point X in source camera u.  K = 4: the bilinear
// footprint around the projection (TL corner i0, j0 and the weight factors
// ax = (1-fx, fx), ay = (1-fy, fy)); K = 1: the token (i0, j0) containing
// the projection.  Returns false when no tap can be inside the image.
struct Footprint {
    int i0, j0;
    float ax[2], ay[2];
};

template <int K>
__device__ __forceinline__ bool footprint(const geocache_camera& cam, float X0, float X1, float X2, int H, int W,
                                          Footprint& f) {
    float uu, vv;
    if (!project(cam, X0, X1, X2, uu, vv)) return false;
    if (K == 1) {
        if (!(uu >= 0.0f && uu < (float)W && vv >= 0.0f && vv < (float)H)) return false;
        f.i0 = (int)floorf(uu);
        f.j0 = (int)floorf(vv);
        f.ax[0] = f.ax[1] = f.ay[0] = f.ay[1] = 1.0f;
        return true;
    }
    const float x = __fsub_rn(uu, 0.5f), y = __fsub_rn(vv, 0.5f);
    if (!(x >= -1.0f && x < (float)W && y >= -1.0f && y < (float)H)) return false;
    const float i0f = floorf(x), j0f = floorf(y);
    f.i0 = (int)i0f;
    f.j0 = (int)j0f;
    const float fx = __fsub_rn(x, i0f), fy = __fsub_rn(y, j0f);
    f.ax[0] = __fsub_rn(1.0f, fx);
    f.ax[1] = fx;
    f.ay[0] = __fsub_rn(1.0f, fy);
    f.ay[1] = fy;
    return true;
}

// Per-tap tests: inside the image, non-zero weight factors, foreground
// texel, ||P_u(q) - X||^2 <= tau2.  Returns the keep mask (bit k = tap k,
// taps ordered TL, TR, BL, BR).  A tap's position is loaded beside its
// validity rather than after it (a background texel's position is read and
// ignored), so the tests wait on one round of loads, not two.
template <int K>
__device__ __forceinline__ int tap_mask(const Footprint& f, const float* __restrict__ pos_u,
                                        const uint8_t* __restrict__ valid_u, int H, int W, float X0, float X1,
                                        float X2, float tau2) {
    int mask = 0;
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const int di = k & 1, dj = k >> 1;
        const int col = f.i0 + di, row = f.j0 + dj;
        if (col < 0 || col >= W || row < 0 || row >= H) continue;
        if (K == 4 && (f.ax[di] == 0.0f || f.ay[dj] == 0.0f)) continue;
        const int q = row * W + col;
        const int fg = __ldg(valid_u + q) != 0;
        const int near = sqdist(pos_u + 3 * (size_t)q, X0, X1, X2) <= tau2;
        mask |= (fg & near) << k;
    }
    return mask;
}

// Indices and renormalised weights of the kept taps of a footprint.
template <int K>
__device__ __forceinline__ void taps_from_mask(const Footprint& f, int mask, int W, Taps& t) {
    taps_clear(t);
    if (!mask) return;
    if (K == 1) {
        t.q[0] = f.j0 * W + f.i0;
        t.w[0] = 1.0f;
        t.kept = 1;
        return;
    }
    float raw[4];
    float sum = 0.0f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        raw[k] = 0.0f;
        if (!((mask >> k) & 1)) continue;
        const int di = k & 1, dj = k >> 1;
        raw[k] = __fmul_rn(f.ax[di], f.ay[dj]);
        t.q[k] = (f.j0 + dj) * W + (f.i0 + di);
        sum = __fadd_rn(sum, raw[k]);
        ++t.kept;
    }
    const float rs = __frcp_rn(sum);
#pragma unroll
    for (int k = 0; k < 4; ++k)
        if (t.q[k] >= 0) t.w[k] = __fmul_rn(raw[k], rs);
}

// The same indices and weights from a sparse record (top-left tap q_tl and the
// footprint fractions fx, fy stored by the build): ax = (1-fx, fx),
// ay = (1-fy, fy) are recomputed exactly as footprint() forms them.
template <int K>
__device__ __forceinline__ void taps_from_record(int mask, int q_tl, float fx, float fy, int W, Taps& t) {
    Footprint f;
    f.ax[0] = __fsub_rn(1.0f, fx);
    f.ax[1] = fx;
    f.ay[0] = __fsub_rn(1.0f, fy);
    f.ay[1] = fy;
    // i0 + j0*W = q_tl; taps_from_mask only uses (j0 + dj)*W + (i0 + di)
    f.i0 = q_tl;
    f.j0 = 0;
    taps_from_mask<K>(f, mask, W, t);
}

// Taps of target point X in source view u (pos_u [H*W*3], valid_u [H*W]):
// footprint, per-tap tests, renormalised weights.  *mask_out (optional)
// receives the keep mask.
template <int K>
__device__ __forceinline__ void compute_taps(const geocache_camera& cam, const float* __restrict__ pos_u,
                                             const uint8_t* __restrict__ valid_u, int H, int W,
                                             float X0, float X1, float X2, float tau2, Taps& t,
                                             int* mask_out = nullptr) {
    Footprint f;
    int mask = 0;
    if (footprint<K>(cam, X0, X1, X2, H, W, f)) mask = tap_mask<K>(f, pos_u, valid_u, H, W, X0, X1, X2, tau2);
    taps_from_mask<K>(f, mask, W, t);
    if (mask_out) *mask_out = mask;
}

}  // namespace geocache
