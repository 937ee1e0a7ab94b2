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
// One thread per quad of 4 consecutive tokens of one view (asset b, view v),
// all channels in groups of 4.  For each group the thread issues 16-byte
// loads of x0 (the anchor's fresh x0, or x0(t-1)) and of x_t first, then for
// views outside the anchor set adds to each covered token the mean over the
// covering anchors of the tap-weighted anchor increments (Eq. 1 with the
// multi-anchor aggregation of Sec. 3.2; uncovered tokens keep x0(t-1)), then
// stores x0(t) and the sampler reconstruction of every token.
// Taps come from the keep masks (MODE = GEOCACHE_CORR_MASK: projection and
// weights recomputed only for covered (token, anchor) pairs), from the full
// per-tap tests (GEOMETRY) or from the tables (TABLE); all three are
// bit-identical.  Streamed rows use evict-first hints so that the anchors'
// rows, which the gathers re-read, stay in L2.
constexpr int kThreads = 256;

template <typename T>
struct Lat4;
template <>
struct Lat4<float> {
    using Raw = float4;
    __device__ static Raw load_raw(const float* p, size_t e, int cnt, bool vec) {
        if (vec) return __ldcs(reinterpret_cast<const float4*>(p + e));
        float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
        if (cnt > 0) r.x = __ldcs(p + e);
        if (cnt > 1) r.y = __ldcs(p + e + 1);
        if (cnt > 2) r.z = __ldcs(p + e + 2);
        if (cnt > 3) r.w = __ldcs(p + e + 3);
        return r;
    }
    __device__ static void unpack(const Raw& x, float (&r)[4]) { r[0] = x.x; r[1] = x.y; r[2] = x.z; r[3] = x.w; }
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
    using Raw = uint2;
    __device__ static Raw load_raw(const __nv_bfloat16* p, size_t e, int cnt, bool vec) {
        if (vec) return __ldcs(reinterpret_cast<const uint2*>(p + e));
        const unsigned short* q = reinterpret_cast<const unsigned short*>(p + e);
        uint32_t h[4] = {0, 0, 0, 0};
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (i < cnt) h[i] = q[i];
        return make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16));
    }
    __device__ static void unpack(const Raw& x, float (&r)[4]) {
        r[0] = __uint_as_float(x.x << 16);
        r[1] = __uint_as_float(x.x & 0xffff0000u);
        r[2] = __uint_as_float(x.y << 16);
        r[3] = __uint_as_float(x.y & 0xffff0000u);
    }
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

// the anchors' rows stay cached (they are re-read by the gathers)
__device__ __forceinline__ void f4_load_keep(const float* p, size_t e, int cnt, bool vec, float (&r)[4]) {
    if (vec) {
        const float4 x = __ldg(reinterpret_cast<const float4*>(p + e));
        r[0] = x.x; r[1] = x.y; r[2] = x.z; r[3] = x.w;
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) r[i] = i < cnt ? __ldg(p + e + i) : 0.0f;
    }
}

// Keep masks of the quad's tokens for source view u, one byte per token.
__device__ __forceinline__ uint32_t quad_masks(const uint8_t* row, int cnt, bool vec) {
    if (vec) return __ldg(reinterpret_cast<const uint32_t*>(row));
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i)
        if (i < cnt) m |= (uint32_t)__ldg(row + i) << (8 * i);
    return m;
}

template <typename T, int K, int MODE, bool VEC>
__global__ void __launch_bounds__(kThreads) transport_quad_kernel(const TransportArgs args) {
    const int HW = args.H * args.W;
    const int p0 = 4 * (blockIdx.x * kThreads + threadIdx.x);
    if (p0 >= HW) return;
    const int cnt = HW - p0 < 4 ? HW - p0 : 4;
    const int v = blockIdx.y, b = blockIdx.z;
    const int N = args.N, C = args.C, a = args.a;
    const int slot = args.slot_of[v];
    const size_t plane = (size_t)HW;
    const size_t view_base = ((size_t)b * N + v) * C * plane + p0;   // element (b, v, 0, p0)
    const bool recon = args.coef.enabled;
    const T* xt_p = static_cast<const T*>(args.x_t);
    T* xn_p = static_cast<T*>(args.x_next);
    const size_t tv = ((size_t)b * N + v) * plane + p0;              // token p0 of (b, v)

    // which of the quad's tokens have any kept tap (any anchor)
    uint32_t any_cover = 0;
    float tau2 = 0.0f;
    if (slot < 0) {
        if (MODE == GEOCACHE_CORR_MASK) {
            const uint8_t* krow = args.keep + ((size_t)b * N + v) * N * plane + p0;
            for (int s = 0; s < a; ++s) any_cover |= quad_masks(krow + (size_t)args.anchors[s] * plane, cnt, VEC);
        } else if (MODE == GEOCACHE_CORR_GEOMETRY) {
            any_cover = quad_masks(args.valid + tv, cnt, VEC);
            const float tu = __ldg(args.tau + b);
            tau2 = __fmul_rn(tu, tu);
        } else {
            any_cover = 0x01010101u;  // tables: every token is looked up
        }
    }

    for (int cg = 0; cg < C; cg += 4) {
        const int cn = C - cg < 4 ? C - cg : 4;
        float x0[4][4];
        typename Lat4<T>::Raw xt[4];
        // streaming loads of the channel group first
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            if (c >= cn) break;
            const size_t e = view_base + (size_t)(cg + c) * plane;
            if (slot >= 0)
                f4_load_keep(args.x0_new, (((size_t)b * a + slot) * C + cg + c) * plane + p0, cnt, VEC, x0[c]);
            else
                Lat4<float>::load(args.x0_prev, e, cnt, VEC, x0[c]);
            if (recon) xt[c] = Lat4<T>::load_raw(xt_p, e, cnt, VEC);
        }
        if (slot < 0) {
            if (any_cover) {
#pragma unroll 1
                for (int i = 0; i < 4; ++i) {
                    if (!((any_cover >> (8 * i)) & 0xff)) continue;
                    const int p = p0 + i;
                    float X0 = 0.f, X1 = 0.f, X2 = 0.f;
                    if (MODE != GEOCACHE_CORR_TABLE) {
                        X0 = __ldg(args.pos + 3 * (tv + i));
                        X1 = __ldg(args.pos + 3 * (tv + i) + 1);
                        X2 = __ldg(args.pos + 3 * (tv + i) + 2);
                    }
                    float acc[4] = {0.f, 0.f, 0.f, 0.f};
                    int n = 0;
                    for (int s = 0; s < a; ++s) {
                        const int u = args.anchors[s];
                        Taps tp;
                        if (MODE == GEOCACHE_CORR_TABLE) {
                            const size_t row = (((size_t)b * N + v) * N + u) * plane + p;
                            tp.kept = 0;
#pragma unroll
                            for (int k = 0; k < K; ++k) {
                                tp.q[k] = __ldg(args.idx + row * K + k);
                                tp.w[k] = __ldg(args.w + row * K + k);
                                tp.kept += tp.q[k] >= 0;
                            }
                        } else {
                            const geocache_camera& cam = args.cams[(size_t)b * N + u];
                            if (MODE == GEOCACHE_CORR_MASK) {
                                const int m = __ldg(args.keep + (((size_t)b * N + v) * N + u) * plane + p);
                                if (!m) continue;
                                Footprint f;
                                footprint<K>(cam, X0, X1, X2, args.H, args.W, f);
                                taps_from_mask<K>(f, m, args.W, tp);
                            } else {
                                const size_t su = ((size_t)b * N + u) * plane;
                                compute_taps<K>(cam, args.pos + 3 * su, args.valid + su, args.H, args.W, X0, X1, X2,
                                                tau2, tp);
                            }
                        }
                        if (!tp.kept) continue;
                        ++n;
                        const float* xn = args.x0_new + (((size_t)b * a + s) * C + cg) * plane;
                        const float* xp = args.x0_prev + (((size_t)b * N + u) * C + cg) * plane;
#pragma unroll
                        for (int k = 0; k < K; ++k) {
                            if (tp.q[k] < 0) continue;
#pragma unroll
                            for (int c = 0; c < 4; ++c) {
                                if (c >= cn) break;
                                const size_t e = (size_t)c * plane + tp.q[k];
                                acc[c] = __fmaf_rn(tp.w[k], __fsub_rn(__ldg(xn + e), __ldg(xp + e)), acc[c]);
                            }
                        }
                    }
                    if (n) {
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const float g = n == 1 ? acc[c] : __fdiv_rn(acc[c], (float)n);
#pragma unroll
                            for (int ii = 0; ii < 4; ++ii)
                                if (ii == i) x0[c][ii] = __fadd_rn(x0[c][ii], g);
                        }
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (c >= cn) break;
                Lat4<float>::store(args.x0_out, view_base + (size_t)(cg + c) * plane, cnt, VEC, x0[c]);
            }
        } else if (args.write_anchor_rows) {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (c >= cn) break;
                Lat4<float>::store(args.x0_out, view_base + (size_t)(cg + c) * plane, cnt, VEC, x0[c]);
            }
        }
        if (recon) {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (c >= cn) break;
                float x[4], y[4], pr[4];
                Lat4<T>::unpack(xt[c], x);
#pragma unroll
                for (int i = 0; i < 4; ++i) y[i] = recon_one(args.coef, x[i], x0[c][i], pr[i]);
                const size_t e = view_base + (size_t)(cg + c) * plane;
                Lat4<T>::store(xn_p, e, cnt, VEC, y);
                if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, VEC, pr);
            }
        }
    }
}

template <typename T, int K, int MODE>
static cudaError_t launch_quad(const TransportArgs& t, cudaStream_t s) {
    const int HW = t.H * t.W;
    const uintptr_t al = (uintptr_t)t.x0_new | (uintptr_t)t.x0_prev | (uintptr_t)t.x0_out | (uintptr_t)t.x_t |
                         (uintptr_t)t.x_next | (uintptr_t)t.pred_out | (uintptr_t)t.keep | (uintptr_t)t.valid;
    const bool vec = (HW % 4 == 0) && (al % 16 == 0);
    const int quads = (HW + 3) / 4;
    dim3 grid((quads + kThreads - 1) / kThreads, t.N, t.B);
    if (vec)
        transport_quad_kernel<T, K, MODE, true><<<grid, kThreads, 0, s>>>(t);
    else
        transport_quad_kernel<T, K, MODE, false><<<grid, kThreads, 0, s>>>(t);
    return cudaGetLastError();
}

template <typename T, int K>
static cudaError_t launch_transport_t(const TransportArgs& t, cudaStream_t s) {
    switch (t.mode) {
        case GEOCACHE_CORR_MASK: return launch_quad<T, K, GEOCACHE_CORR_MASK>(t, s);
        case GEOCACHE_CORR_TABLE: return launch_quad<T, K, GEOCACHE_CORR_TABLE>(t, s);
        default: return launch_quad<T, K, GEOCACHE_CORR_GEOMETRY>(t, s);
    }
}

int transport_launch_count(int, int, int in_place) { return 1 + (in_place ? 1 : 0); }

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
