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
// One thread per (asset b, target view v, source view u, token p).
template <int K>
__global__ void __launch_bounds__(256) build_corr_kernel(const float* __restrict__ pos,
                                                         const uint8_t* __restrict__ valid,
                                                         const geocache_camera* __restrict__ cams,
                                                         const float* __restrict__ tau, int N, int H, int W,
                                                         int32_t* __restrict__ idx, float* __restrict__ wout) {
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
    const size_t tv = ((size_t)b * N + v) * HW + p;
    if (u != v && __ldg(valid + tv)) {
        const float tu = __ldg(tau + b);
        const size_t su = ((size_t)b * N + u) * HW;
        compute_taps<K>(s_cam, pos + 3 * su, valid + su, H, W, __ldg(pos + 3 * tv), __ldg(pos + 3 * tv + 1),
                        __ldg(pos + 3 * tv + 2), __fmul_rn(tu, tu), t);
    }
    const size_t row = (((size_t)b * N + v) * N + u) * HW + p;
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
        build_corr_kernel<4><<<grid, 256, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W, c.idx, c.w);
    else
        build_corr_kernel<1><<<grid, 256, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W, c.idx, c.w);
    return cudaGetLastError();
}

// ------------------------------------------------- fused transport step --
// One thread per (asset b, view v, token p), channels [c0, c0+cn) with
// cn <= CMAX.  Anchor views take the denoiser's x0; other views add the mean
// over covering anchors of the tap-weighted anchor increments (Eq. 1), then
// every view is reconstructed (Sec. 3.2).
template <typename T, int K, int CMAX>
__global__ void __launch_bounds__(256) transport_kernel(const TransportArgs args) {
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
        if (fg && args.mode == GEOCACHE_CORR_GEOMETRY) {
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

template <typename T, int K>
static cudaError_t launch_transport_t(const TransportArgs& t, cudaStream_t s) {
    const int HW = t.H * t.W;
    dim3 grid((HW + 255) / 256, t.N, t.B);
    if (t.cn <= 4)
        transport_kernel<T, K, 4><<<grid, 256, 0, s>>>(t);
    else
        transport_kernel<T, K, 16><<<grid, 256, 0, s>>>(t);
    return cudaGetLastError();
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
template <typename T>
__global__ void __launch_bounds__(256) reconstruct_kernel(const T* xt, const float* x0, T* xn, int64_t n,
                                                          const ReconCoef coef, float* pred_out, float* x0_store) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const float x = x0[i];
        float pred;
        const float y = recon_one(coef, lat_load(xt, i), x, pred);
        lat_store(xn, i, y);
        if (pred_out) pred_out[i] = pred;
        if (x0_store) x0_store[i] = x;
    }
}

cudaError_t launch_reconstruct(const void* x_t, const float* x0, void* x_next, int lat_dtype, int64_t n,
                               const ReconCoef& coef, float* pred_out, float* x0_store, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    if (lat_dtype == GEOCACHE_BF16)
        reconstruct_kernel<__nv_bfloat16><<<(unsigned)blocks, 256, 0, s>>>(
            static_cast<const __nv_bfloat16*>(x_t), x0, static_cast<__nv_bfloat16*>(x_next), n, coef, pred_out,
            x0_store);
    else
        reconstruct_kernel<float><<<(unsigned)blocks, 256, 0, s>>>(static_cast<const float*>(x_t), x0,
                                                                    static_cast<float*>(x_next), n, coef,
                                                                    pred_out, x0_store);
    return cudaGetLastError();
}

}  // namespace geocache
