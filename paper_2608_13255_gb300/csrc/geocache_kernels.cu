// CUDA kernels (sm_103a) of the geometric delta transport (GeoCache,
// Sec. 3.2): tau, the correspondence tables, the fused transport +
// reconstruction step, and the full-step reconstruction.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cfloat>
#include <cstdint>

#include "geocache_device.cuh"
#include "geocache_internal.h"

namespace geocache {

// ---------------------------------------------------------------- latents --
__device__ __forceinline__ float lat_load(const float* p, size_t i) { return __ldg(p + i); }
__device__ __forceinline__ float lat_load(const __nv_bfloat16* p, size_t i) {
    return __bfloat162float(p[i]);
}
__device__ __forceinline__ void lat_store(float* p, size_t i, float v) { p[i] = v; }
__device__ __forceinline__ void lat_store(__nv_bfloat16* p, size_t i, float v) {
    p[i] = __float2bfloat16_rn(v);
}

// Sampler conversion of one element (Sec. 3.2, closed-form relations after
// Eq. 1).  Fixed operation sequence (explicit intrinsics) so that the fused
// transport step and the standalone reconstruction agree bit for bit.
__device__ __forceinline__ float recon_one(const ReconCoef& c, float xt, float x0, float& pred) {
    if (c.sampler == GEOCACHE_DDIM) {
        const float eps = __fmul_rn(__fmaf_rn(-c.st, x0, xt), c.inv_s1t);
        pred = (c.pred_kind == GEOCACHE_PRED_V) ? __fmaf_rn(c.st, eps, -__fmul_rn(c.s1t, x0)) : eps;
        return __fmaf_rn(c.sp, x0, __fmul_rn(c.s1p, eps));
    } else {
        const float vel = __fmul_rn(__fsub_rn(xt, x0), c.inv_sigma);
        pred = vel;
        return __fmaf_rn(c.dsigma, vel, xt);
    }
}

// -------------------------------------------------------------------- tau --
// One CTA per asset: componentwise min / max of the foreground texels of all
// N views (order-free and exact), then tau = tol_frac * sqrt(diag^2) with the
// squares summed ((d0^2 + d1^2) + d2^2) in binary32.
__global__ void __launch_bounds__(1024) tau_kernel(const float* __restrict__ pos,
                                                   const uint8_t* __restrict__ valid, int N, int H,
                                                   int W, float tol_frac, float* __restrict__ tau) {
    const int b = blockIdx.x;
    const size_t per = (size_t)N * H * W;
    const float* P = pos + 3 * per * b;
    const uint8_t* V = valid + per * b;
    float lo[3] = {FLT_MAX, FLT_MAX, FLT_MAX}, hi[3] = {-FLT_MAX, -FLT_MAX, -FLT_MAX};
    int any = 0;
    for (size_t i = threadIdx.x; i < per; i += blockDim.x) {
        if (!V[i]) continue;
        any = 1;
#pragma unroll
        for (int c = 0; c < 3; ++c) {
            const float x = P[3 * i + c];
            lo[c] = fminf(lo[c], x);
            hi[c] = fmaxf(hi[c], x);
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
        for (int c = 0; c < 3; ++c) {
            lo[c] = fminf(lo[c], __shfl_xor_sync(0xffffffffu, lo[c], off));
            hi[c] = fmaxf(hi[c], __shfl_xor_sync(0xffffffffu, hi[c], off));
        }
        any |= __shfl_xor_sync(0xffffffffu, any, off);
    }
    __shared__ float s_lo[32][3], s_hi[32][3];
    __shared__ int s_any[32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
#pragma unroll
        for (int c = 0; c < 3; ++c) { s_lo[warp][c] = lo[c]; s_hi[warp][c] = hi[c]; }
        s_any[warp] = any;
    }
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
#pragma unroll
        for (int c = 0; c < 3; ++c) {
            lo[c] = lane < nw ? s_lo[lane][c] : FLT_MAX;
            hi[c] = lane < nw ? s_hi[lane][c] : -FLT_MAX;
        }
        any = lane < nw ? s_any[lane] : 0;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
            for (int c = 0; c < 3; ++c) {
                lo[c] = fminf(lo[c], __shfl_xor_sync(0xffffffffu, lo[c], off));
                hi[c] = fmaxf(hi[c], __shfl_xor_sync(0xffffffffu, hi[c], off));
            }
            any |= __shfl_xor_sync(0xffffffffu, any, off);
        }
        if (lane == 0) {
            float t = 0.0f;
            if (any) {
                const float d0 = __fsub_rn(hi[0], lo[0]), d1 = __fsub_rn(hi[1], lo[1]),
                            d2 = __fsub_rn(hi[2], lo[2]);
                const float diag2 =
                    __fadd_rn(__fadd_rn(__fmul_rn(d0, d0), __fmul_rn(d1, d1)), __fmul_rn(d2, d2));
                t = __fmul_rn(tol_frac, __fsqrt_rn(diag2));
            }
            tau[b] = t;
        }
    }
}

cudaError_t launch_tau(const float* pos, const uint8_t* valid, int B, int N, int H, int W, float tol_frac,
                       float* tau, cudaStream_t s) {
    tau_kernel<<<B, 1024, 0, s>>>(pos, valid, N, H, W, tol_frac, tau);
    return cudaGetLastError();
}

// ------------------------------------------------------- correspondence --
// One thread per (asset b, target view v, source view u, token p): the
// tables idx/w (when non-NULL) and the keep masks (when non-NULL).
template <int K>
__global__ void __launch_bounds__(256) build_corr_kernel(const float* __restrict__ pos,
                                                         const uint8_t* __restrict__ valid,
                                                         const geocache_camera* __restrict__ cams,
                                                         const float* __restrict__ tau, int N, int H, int W,
                                                         int32_t* __restrict__ idx, float* __restrict__ wout,
                                                         uint8_t* __restrict__ keep) {
    const int HW = H * W;
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    const int v = blockIdx.y / N, u = blockIdx.y % N, b = blockIdx.z;
    __shared__ geocache_camera s_cam;
    if (threadIdx.x < 16) reinterpret_cast<float*>(&s_cam)[threadIdx.x] =
        __ldg(reinterpret_cast<const float*>(cams + (size_t)b * N + u) + threadIdx.x);
    __syncthreads();
    if (p >= HW) return;
    Taps t;
    taps_clear(t);
    int mask = 0;
    const size_t tv = ((size_t)b * N + v) * HW + p;
    if (u != v && __ldg(valid + tv)) {
        const float tu = __ldg(tau + b);
        const size_t su = ((size_t)b * N + u) * HW;
        compute_taps<K>(s_cam, pos + 3 * su, valid + su, H, W, __ldg(pos + 3 * tv), __ldg(pos + 3 * tv + 1),
                        __ldg(pos + 3 * tv + 2), __fmul_rn(tu, tu), t, &mask);
    }
    const size_t row = (((size_t)b * N + v) * N + u) * HW + p;
    if (keep) keep[row] = (uint8_t)mask;
    if (!idx) return;
    if (K == 4) {
        reinterpret_cast<int4*>(idx)[row] = make_int4(t.q[0], t.q[1], t.q[2], t.q[3]);
        reinterpret_cast<float4*>(wout)[row] = make_float4(t.w[0], t.w[1], t.w[2], t.w[3]);
    } else {
        idx[row] = t.q[0];
        wout[row] = t.w[0];
    }
}

cudaError_t launch_build_corr(const geocache_corr& c, cudaStream_t s) {
    const int HW = c.H * c.W;
    dim3 grid((HW + 255) / 256, c.N * c.N, c.B);
    if (c.K == 4)
        build_corr_kernel<4><<<grid, 256, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W, c.idx, c.w, c.keep);
    else
        build_corr_kernel<1><<<grid, 256, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W, c.idx, c.w, c.keep);
    return cudaGetLastError();
}

// ------------------------------------------------- fused transport step --
// General variant (any number of anchors): one thread per (asset b, view v,
// token p), channels [c0, c0+cn) with cn <= CMAX.  Anchor views take the
// denoiser's x0; other views add the mean over covering anchors of the
// tap-weighted anchor increments (Eq. 1), then every view is reconstructed
// (Sec. 3.2).
template <typename T, int K, int CMAX>
__global__ void __launch_bounds__(256) transport_pixel_kernel(const TransportArgs args) {
    const int HW = args.H * args.W;
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    const int v = blockIdx.y, b = blockIdx.z;
    if (p >= HW) return;
    const int N = args.N, C = args.C, cn = args.cn, c0 = args.c0;
    const size_t plane0 = (((size_t)b * N + v) * C + c0) * HW + p;  // element (b, v, c0, p)
    const int slot = args.slot_of[v];
    float x0v[CMAX];
    if (slot >= 0) {
        const float* src = args.x0_new + (((size_t)b * args.a + slot) * C + c0) * HW + p;
#pragma unroll
        for (int c = 0; c < CMAX; ++c)
            if (c < cn) x0v[c] = __ldg(src + (size_t)c * HW);
        if (args.write_anchor_rows) {
#pragma unroll
            for (int c = 0; c < CMAX; ++c)
                if (c < cn) args.x0_out[plane0 + (size_t)c * HW] = x0v[c];
        }
    } else {
        float acc[CMAX];
#pragma unroll
        for (int c = 0; c < CMAX; ++c) acc[c] = 0.0f;
        int n = 0;
        const size_t tv = ((size_t)b * N + v) * HW + p;
        const bool fg = (args.mode == GEOCACHE_CORR_TABLE) || __ldg(args.valid + tv);
        float X0 = 0.f, X1 = 0.f, X2 = 0.f, tau2 = 0.f;
        if (fg && args.mode != GEOCACHE_CORR_TABLE) {  // geometry and keep-mask modes recompute the taps
            X0 = __ldg(args.pos + 3 * tv);
            X1 = __ldg(args.pos + 3 * tv + 1);
            X2 = __ldg(args.pos + 3 * tv + 2);
            const float tu = __ldg(args.tau + b);
            tau2 = __fmul_rn(tu, tu);
        }
        if (fg) {
            for (int s = 0; s < args.a; ++s) {
                const int u = args.anchors[s];
                Taps t;
                if (args.mode == GEOCACHE_CORR_TABLE) {
                    const size_t row = (((size_t)b * N + v) * N + u) * HW + p;
                    t.kept = 0;
#pragma unroll
                    for (int k = 0; k < K; ++k) {
                        t.q[k] = __ldg(args.idx + row * K + k);
                        t.w[k] = __ldg(args.w + row * K + k);
                        t.kept += t.q[k] >= 0;
                    }
                } else {
                    const size_t su = ((size_t)b * N + u) * HW;
                    compute_taps<K>(args.cams[(size_t)b * N + u], args.pos + 3 * su, args.valid + su,
                                    args.H, args.W, X0, X1, X2, tau2, t);
                }
                if (!t.kept) continue;
                ++n;
                const float* xn = args.x0_new + (((size_t)b * args.a + s) * C + c0) * HW;
                const float* xp = args.x0_prev + (((size_t)b * N + u) * C + c0) * HW;
#pragma unroll
                for (int c = 0; c < CMAX; ++c) {
                    if (c >= cn) break;
                    float g = 0.0f;
#pragma unroll
                    for (int k = 0; k < K; ++k) {
                        if (t.q[k] < 0) continue;
                        const size_t e = (size_t)c * HW + t.q[k];
                        g = __fmaf_rn(t.w[k], __fsub_rn(__ldg(xn + e), __ldg(xp + e)), g);
                    }
                    acc[c] = __fadd_rn(acc[c], g);
                }
            }
        }
#pragma unroll
        for (int c = 0; c < CMAX; ++c) {
            if (c < cn) {
                const float prev = __ldg(args.x0_prev + plane0 + (size_t)c * HW);
                x0v[c] = n ? __fadd_rn(prev, __fdiv_rn(acc[c], (float)n)) : prev;
                args.x0_out[plane0 + (size_t)c * HW] = x0v[c];
            }
        }
    }
    if (args.coef.enabled) {
        const T* xt = static_cast<const T*>(args.x_t);
        T* xnx = static_cast<T*>(args.x_next);
#pragma unroll
        for (int c = 0; c < CMAX; ++c) {
            if (c < cn) {
                const size_t e = plane0 + (size_t)c * HW;
                float pred;
                const float y = recon_one(args.coef, lat_load(xt, e), x0v[c], pred);
                lat_store(xnx, e, y);
                if (args.pred_out) args.pred_out[e] = pred;
            }
        }
    }
}

// Tiled variant (a <= kTileMaxAnchors), the hot path.  One CTA owns a tile
// of 256 consecutive tokens of one view (asset b, view v) and all channels.
//  phase 0 (views outside the anchor set): thread t finds the kept taps of
//    token 4*(t%64) + t/64 for every anchor and stores them in shared memory
//    at column t, with the number n of covering anchors;
//  phase 1: thread t handles the 4 consecutive tokens 4*(t%64).. of channel
//    t/64 (+4, +8, ... for C > 4): 16-byte loads of x0(t-1) or the anchor's
//    x0 and of x_t (issued before phase 0 so they overlap the geometry), the
//    gathered increment sum_j w_j (x0_new - x0_prev)[q_j] / n, the cache
//    store and the sampler reconstruction.
// Streamed rows use evict-first cache hints so that the anchors' rows, which
// the gathers re-read, stay in L2.
constexpr int kTile = 256;
constexpr int kTileMaxAnchors = 8;

template <typename T>
struct Lat4;
template <>
struct Lat4<float> {
    using V = float4;
    __device__ static void load(const float* p, size_t e, int cnt, bool vec, float (&r)[4]) {
        if (vec) {
            const float4 x = __ldcs(reinterpret_cast<const float4*>(p + e));
            r[0] = x.x; r[1] = x.y; r[2] = x.z; r[3] = x.w;
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) r[i] = i < cnt ? __ldcs(p + e + i) : 0.0f;
        }
    }
    __device__ static void store(float* p, size_t e, int cnt, bool vec, const float (&r)[4]) {
        if (vec) {
            __stcs(reinterpret_cast<float4*>(p + e), make_float4(r[0], r[1], r[2], r[3]));
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (i < cnt) __stcs(p + e + i, r[i]);
        }
    }
};
template <>
struct Lat4<__nv_bfloat16> {
    __device__ static void load(const __nv_bfloat16* p, size_t e, int cnt, bool vec, float (&r)[4]) {
        if (vec) {
            const uint2 x = __ldcs(reinterpret_cast<const uint2*>(p + e));
            const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162*>(&x.x);
            const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162*>(&x.y);
            r[0] = __low2float(lo); r[1] = __high2float(lo); r[2] = __low2float(hi); r[3] = __high2float(hi);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) r[i] = i < cnt ? __bfloat162float(p[e + i]) : 0.0f;
        }
    }
    __device__ static void store(__nv_bfloat16* p, size_t e, int cnt, bool vec, const float (&r)[4]) {
        if (vec) {
            __nv_bfloat162 lo = __floats2bfloat162_rn(r[0], r[1]);
            __nv_bfloat162 hi = __floats2bfloat162_rn(r[2], r[3]);
            uint2 x;
            x.x = *reinterpret_cast<uint32_t*>(&lo);
            x.y = *reinterpret_cast<uint32_t*>(&hi);
            __stcs(reinterpret_cast<uint2*>(p + e), x);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (i < cnt) p[e + i] = __float2bfloat16_rn(r[i]);
        }
    }
};

__device__ __forceinline__ void f4_load(const float* p, size_t e, int cnt, bool vec, float (&r)[4]) {
    Lat4<float>::load(p, e, cnt, vec, r);
}
// anchor rows: keep them in L2 for the gathers (default caching)
__device__ __forceinline__ void f4_load_keep(const float* p, size_t e, int cnt, bool vec, float (&r)[4]) {
    if (vec) {
        const float4 x = __ldg(reinterpret_cast<const float4*>(p + e));
        r[0] = x.x; r[1] = x.y; r[2] = x.z; r[3] = x.w;
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) r[i] = i < cnt ? __ldg(p + e + i) : 0.0f;
    }
}

template <typename T, int K, bool VEC>
__global__ void __launch_bounds__(kTile) transport_tile_kernel(const TransportArgs args) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int HW = args.H * args.W;
    const int tile0 = blockIdx.x * kTile;
    const int v = blockIdx.y, b = blockIdx.z;
    const int N = args.N, C = args.C, a = args.a;
    const int slot = args.slot_of[v];
    const int t = threadIdx.x;
    const int quad = t & 63;
    const int E = K * a;  // tap entries per token
    geocache_camera* s_cam = reinterpret_cast<geocache_camera*>(smem);
    int32_t* s_q = reinterpret_cast<int32_t*>(smem + sizeof(geocache_camera) * kTileMaxAnchors);
    float* s_w = reinterpret_cast<float*>(s_q + E * kTile);
    uint8_t* s_s = reinterpret_cast<uint8_t*>(s_w + E * kTile);
    uint8_t* s_len = s_s + E * kTile;
    uint8_t* s_n = s_len + kTile;

    // phase-1 role and the first channel pass's streaming loads
    const int p0 = tile0 + 4 * quad;
    const int cnt = HW - p0 < 4 ? HW - p0 : 4;
    int c = t >> 6;
    const size_t view_base = ((size_t)b * N + v) * C;
    const size_t anc_base = slot >= 0 ? ((size_t)b * a + slot) * C : 0;
    const bool recon = args.coef.enabled;
    const T* xt_p = static_cast<const T*>(args.x_t);
    float x0[4], xt[4];
    if (cnt > 0 && c < C) {
        if (slot >= 0)
            f4_load_keep(args.x0_new, (anc_base + c) * HW + p0, cnt, VEC, x0);
        else
            f4_load(args.x0_prev, (view_base + c) * HW + p0, cnt, VEC, x0);
        if (recon) Lat4<T>::load(xt_p, (view_base + c) * HW + p0, cnt, VEC, xt);
    }

    if (slot < 0) {
        // ------------------------------------------------------ phase 0 --
        const bool table = args.mode == GEOCACHE_CORR_TABLE;
        if (!table)
            for (int i = t; i < a * 16; i += kTile)
                reinterpret_cast<float*>(s_cam)[i] =
                    __ldg(reinterpret_cast<const float*>(args.cams + (size_t)b * N + args.anchors[i >> 4]) + (i & 15));
        __syncthreads();
        const int p = tile0 + 4 * (t & 63) + (t >> 6);
        int len = 0, n = 0;
        if (p < HW) {
            const size_t tv = ((size_t)b * N + v) * HW + p;
            if (table) {
                for (int s = 0; s < a; ++s) {
                    const size_t row = (((size_t)b * N + v) * N + args.anchors[s]) * HW + p;
                    int kept = 0;
#pragma unroll
                    for (int k = 0; k < K; ++k) {
                        const int32_t q = __ldg(args.idx + row * K + k);
                        if (q >= 0) {
                            s_q[len * kTile + t] = q;
                            s_w[len * kTile + t] = __ldg(args.w + row * K + k);
                            s_s[len * kTile + t] = (uint8_t)s;
                            ++len;
                            ++kept;
                        }
                    }
                    n += kept > 0;
                }
            } else if (args.mode == GEOCACHE_CORR_MASK) {
                // keep masks of every anchor first (independent byte loads), then
                // the projection and weights only for the covering anchors
                const uint8_t* krow = args.keep + ((size_t)b * N + v) * N * HW + p;
                uint32_t masks = 0;
                for (int s = 0; s < a; ++s) masks |= (uint32_t)__ldg(krow + (size_t)args.anchors[s] * HW) << (4 * s);
                if (masks) {
                    const float X0 = __ldg(args.pos + 3 * tv), X1 = __ldg(args.pos + 3 * tv + 1),
                                X2 = __ldg(args.pos + 3 * tv + 2);
                    for (int s = 0; s < a; ++s) {
                        const int m = (masks >> (4 * s)) & 15;
                        if (!m) continue;
                        Footprint f;
                        footprint<K>(s_cam[s], X0, X1, X2, args.H, args.W, f);
                        Taps tp;
                        taps_from_mask<K>(f, m, args.W, tp);
                        ++n;
#pragma unroll
                        for (int k = 0; k < K; ++k) {
                            if (tp.q[k] < 0) continue;
                            s_q[len * kTile + t] = tp.q[k];
                            s_w[len * kTile + t] = tp.w[k];
                            s_s[len * kTile + t] = (uint8_t)s;
                            ++len;
                        }
                    }
                }
            } else if (__ldg(args.valid + tv)) {
                const float X0 = __ldg(args.pos + 3 * tv), X1 = __ldg(args.pos + 3 * tv + 1),
                            X2 = __ldg(args.pos + 3 * tv + 2);
                const float tu = __ldg(args.tau + b);
                const float tau2 = __fmul_rn(tu, tu);
                for (int s = 0; s < a; ++s) {
                    const size_t su = ((size_t)b * N + args.anchors[s]) * HW;
                    Taps tp;
                    compute_taps<K>(s_cam[s], args.pos + 3 * su, args.valid + su, args.H, args.W, X0, X1, X2, tau2,
                                    tp);
                    if (!tp.kept) continue;
                    ++n;
#pragma unroll
                    for (int k = 0; k < K; ++k) {
                        if (tp.q[k] < 0) continue;
                        s_q[len * kTile + t] = tp.q[k];
                        s_w[len * kTile + t] = tp.w[k];
                        s_s[len * kTile + t] = (uint8_t)s;
                        ++len;
                    }
                }
            }
        }
        s_len[t] = (uint8_t)len;
        s_n[t] = (uint8_t)n;
        __syncthreads();
    }

    // ---------------------------------------------------------- phase 1 --
    if (cnt <= 0) return;
    T* xn_p = static_cast<T*>(args.x_next);
    for (; c < C; c += 4) {
        const size_t e = (view_base + c) * HW + p0;
        if (slot < 0) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int col = i * 64 + quad;
                const int n = s_n[col];
                if (!n) continue;
                const int len = s_len[col];
                float acc = 0.0f;
                for (int j = 0; j < len; ++j) {
                    const int q = s_q[j * kTile + col];
                    const float wj = s_w[j * kTile + col];
                    const int s = s_s[j * kTile + col];
                    const float xn = __ldg(args.x0_new + (((size_t)b * a + s) * C + c) * HW + q);
                    const float xp = __ldg(args.x0_prev + (((size_t)b * N + args.anchors[s]) * C + c) * HW + q);
                    acc = __fmaf_rn(wj, __fsub_rn(xn, xp), acc);
                }
                x0[i] = __fadd_rn(x0[i], __fdiv_rn(acc, (float)n));
            }
            Lat4<float>::store(args.x0_out, e, cnt, VEC, x0);
        } else if (args.write_anchor_rows) {
            Lat4<float>::store(args.x0_out, e, cnt, VEC, x0);
        }
        if (recon) {
            float y[4], pr[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) y[i] = recon_one(args.coef, xt[i], x0[i], pr[i]);
            Lat4<T>::store(xn_p, e, cnt, VEC, y);
            if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, VEC, pr);
        }
        if (c + 4 < C) {
            if (slot >= 0)
                f4_load_keep(args.x0_new, (anc_base + c + 4) * HW + p0, cnt, VEC, x0);
            else
                f4_load(args.x0_prev, (view_base + c + 4) * HW + p0, cnt, VEC, x0);
            if (recon) Lat4<T>::load(xt_p, (view_base + c + 4) * HW + p0, cnt, VEC, xt);
        }
    }
}

size_t tile_smem_bytes(int K, int a) {
    return sizeof(geocache_camera) * kTileMaxAnchors + (size_t)K * a * kTile * 9 + 2 * kTile;
}

template <typename T, int K>
static cudaError_t launch_transport_t(const TransportArgs& t, cudaStream_t s) {
    const int HW = t.H * t.W;
    if (t.a <= kTileMaxAnchors) {
        const uintptr_t al = (uintptr_t)t.x0_new | (uintptr_t)t.x0_prev | (uintptr_t)t.x0_out |
                             (uintptr_t)t.x_t | (uintptr_t)t.x_next | (uintptr_t)t.pred_out;
        const bool vec = (HW % 4 == 0) && (al % 16 == 0);
        const size_t smem = tile_smem_bytes(K, t.a);
        dim3 grid((HW + kTile - 1) / kTile, t.N, t.B);
        auto kern = vec ? transport_tile_kernel<T, K, true> : transport_tile_kernel<T, K, false>;
        if (smem > 48 * 1024) {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
        kern<<<grid, kTile, smem, s>>>(t);
        return cudaGetLastError();
    }
    dim3 grid((HW + 255) / 256, t.N, t.B);
    TransportArgs c = t;
    const int chunk = t.C <= 4 ? 4 : 16;
    for (int c0 = 0; c0 < t.C; c0 += chunk) {
        c.c0 = c0;
        c.cn = t.C - c0 < chunk ? t.C - c0 : chunk;
        if (c.cn <= 4)
            transport_pixel_kernel<T, K, 4><<<grid, 256, 0, s>>>(c);
        else
            transport_pixel_kernel<T, K, 16><<<grid, 256, 0, s>>>(c);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

int transport_launch_count(int a, int C, int in_place) {
    int n = a <= kTileMaxAnchors ? 1 : (C + (C <= 4 ? 4 : 16) - 1) / (C <= 4 ? 4 : 16);
    return n + (in_place ? 1 : 0);
}

cudaError_t launch_transport(const TransportArgs& t, cudaStream_t s) {
    if (t.lat_dtype == GEOCACHE_BF16)
        return t.K == 4 ? launch_transport_t<__nv_bfloat16, 4>(t, s) : launch_transport_t<__nv_bfloat16, 1>(t, s);
    return t.K == 4 ? launch_transport_t<float, 4>(t, s) : launch_transport_t<float, 1>(t, s);
}

// Anchors' rows of an in-place cache update, written after the gathers.
__global__ void copy_anchor_rows_kernel(const TransportArgs args) {
    const size_t HW = (size_t)args.H * args.W;
    const size_t per = (size_t)args.cn * HW;
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int s = blockIdx.y, b = blockIdx.z;
    if (i >= per) return;
    const int u = args.anchors[s];
    args.x0_out[(((size_t)b * args.N + u) * args.C + args.c0) * HW + i] =
        args.x0_new[(((size_t)b * args.a + s) * args.C + args.c0) * HW + i];
}

cudaError_t launch_copy_anchor_rows(const TransportArgs& t, cudaStream_t s) {
    const size_t per = (size_t)t.cn * t.H * t.W;
    dim3 grid((unsigned)((per + 255) / 256), t.a, t.B);
    copy_anchor_rows_kernel<<<grid, 256, 0, s>>>(t);
    return cudaGetLastError();
}

// ---------------------------------------------------- full-step recon --
// Elementwise x_t, x0 -> x_next (and optionally pred, a copy of x0), four
// consecutive elements per thread with 16-byte accesses when every pointer
// is 16-byte aligned; grid-stride over groups of four.
template <typename T, bool VEC>
__global__ void __launch_bounds__(256) reconstruct_kernel(const T* xt, const float* x0, T* xn, int64_t n,
                                                          const ReconCoef coef, float* pred_out, float* x0_store) {
    const int64_t groups = (n + 3) / 4;
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups;
         g += (int64_t)gridDim.x * blockDim.x) {
        const int64_t e = 4 * g;
        const int cnt = n - e < 4 ? (int)(n - e) : 4;
        const bool vec = VEC && cnt == 4;
        float a[4], x[4], y[4], pr[4];
        Lat4<float>::load(x0, e, cnt, vec, a);
        Lat4<T>::load(xt, e, cnt, vec, x);
#pragma unroll
        for (int i = 0; i < 4; ++i) y[i] = recon_one(coef, x[i], a[i], pr[i]);
        Lat4<T>::store(xn, e, cnt, vec, y);
        if (pred_out) Lat4<float>::store(pred_out, e, cnt, vec, pr);
        if (x0_store) Lat4<float>::store(x0_store, e, cnt, vec, a);
    }
}

template <typename T>
static cudaError_t launch_reconstruct_t(const void* x_t, const float* x0, void* x_next, int64_t n,
                                        const ReconCoef& coef, float* pred_out, float* x0_store, cudaStream_t s) {
    int64_t blocks = ((n + 3) / 4 + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    const uintptr_t al = (uintptr_t)x_t | (uintptr_t)x0 | (uintptr_t)x_next | (uintptr_t)pred_out | (uintptr_t)x0_store;
    const T* xt = static_cast<const T*>(x_t);
    T* xn = static_cast<T*>(x_next);
    if (al % 16 == 0)
        reconstruct_kernel<T, true><<<(unsigned)blocks, 256, 0, s>>>(xt, x0, xn, n, coef, pred_out, x0_store);
    else
        reconstruct_kernel<T, false><<<(unsigned)blocks, 256, 0, s>>>(xt, x0, xn, n, coef, pred_out, x0_store);
    return cudaGetLastError();
}

cudaError_t launch_reconstruct(const void* x_t, const float* x0, void* x_next, int lat_dtype, int64_t n,
                               const ReconCoef& coef, float* pred_out, float* x0_store, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if (lat_dtype == GEOCACHE_BF16)
        return launch_reconstruct_t<__nv_bfloat16>(x_t, x0, x_next, n, coef, pred_out, x0_store, s);
    return launch_reconstruct_t<float>(x_t, x0, x_next, n, coef, pred_out, x0_store, s);
}

}  // namespace geocache
