// CUDA kernels (sm_103a) of the geometric delta transport (GeoCache,
// Sec. 3.2): tau, the correspondence tables, the fused transport +
// reconstruction step, and the full-step reconstruction.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cooperative_groups.h>

#include <atomic>
#include <cfloat>
#include <cstdint>

#include "geocache_device.cuh"
#include "geocache_internal.h"

namespace geocache {

__host__ __device__ int tiles_per_view(int H, int W) { return (H * W + GEOCACHE_TILE_TOKENS - 1) / GEOCACHE_TILE_TOKENS; }

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

// One kept tap's term of an anchor's transported quantity, accumulated in
// tap order: Eq. 1 carries the anchor's change x0_new - x0(t-1); the
// value-copy ablation (Sec. 4.3, "delta -> copy") carries x0_new itself.
__device__ __forceinline__ float tap_term(bool copy, float w, float xn, float xp, float acc) {
    return __fmaf_rn(w, copy ? xn : __fsub_rn(xn, xp), acc);
}

// x0(t) of a covered target from x0(t-1) and the anchor-ordered sum g of its
// n covering anchors' terms: x0 + g/n (Eq. 1, normalised multi-anchor sum),
// or g/n under the value copy.
__device__ __forceinline__ float fold_one(bool copy, float x0, float g, int n) {
    // g / n correctly rounded; for n a power of two that is exactly g * (1 / n)
    const float m = n == 1 ? g
                           : ((n & (n - 1)) == 0 ? __fmul_rn(g, __frcp_rn((float)n)) : __fdiv_rn(g, (float)n));
    return copy ? m : __fadd_rn(x0, m);
}

// -------------------------------------------------------------------- tau --
// One thread-block cluster per asset: CTA r of the cluster reduces the
// componentwise min / max of the foreground texels of slice r of the asset's
// texels (exact and order-free), the cluster combines the partial boxes through
// distributed shared memory, and CTA 0 writes tau = tol_frac * sqrt(diag^2)
// with the squares summed ((d0^2 + d1^2) + d2^2) in binary32.
struct Box {
    float lo[3], hi[3];
    int any;
};

__device__ __forceinline__ void box_reduce_warp(Box& x) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
        for (int c = 0; c < 3; ++c) {
            x.lo[c] = fminf(x.lo[c], __shfl_xor_sync(0xffffffffu, x.lo[c], off));
            x.hi[c] = fmaxf(x.hi[c], __shfl_xor_sync(0xffffffffu, x.hi[c], off));
        }
        x.any |= __shfl_xor_sync(0xffffffffu, x.any, off);
    }
}

__global__ void __launch_bounds__(256, 8) tau_kernel(const float* __restrict__ pos, const uint8_t* __restrict__ valid,
                                                     int N, int HW, float tol_frac, int quads, float* __restrict__ tau) {
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    const int cs = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const int b = blockIdx.x / cs;
    __shared__ Box s_warp[16];
    __shared__ Box s_part;
    Box x;
#pragma unroll
    for (int c = 0; c < 3; ++c) { x.lo[c] = FLT_MAX; x.hi[c] = -FLT_MAX; }
    x.any = 0;
    // the asset's N views are contiguous: each CTA of the cluster takes one
    // slice of their N * HW texels
    const size_t n = (size_t)N * HW;
    const size_t base = (size_t)b * n;
    if (quads) {  // four texels per load: their 4 validity bytes and 12 position floats
        const size_t nq = n / 4, per = (nq + cs - 1) / cs;
        const size_t q0 = (size_t)rank * per, q1 = q0 + per < nq ? q0 + per : nq;
        const uint32_t* vq = reinterpret_cast<const uint32_t*>(valid + base);
        const float4* pq = reinterpret_cast<const float4*>(pos + 3 * base);
#pragma unroll 4
        for (size_t i = q0 + threadIdx.x; i < q1; i += blockDim.x) {
            const uint32_t m = __ldg(vq + i);
            if (!m) continue;  // background quads: their positions are not read
            x.any = 1;
            const float4 f0 = __ldg(pq + 3 * i), f1 = __ldg(pq + 3 * i + 1), f2 = __ldg(pq + 3 * i + 2);
            const float f[12] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w, f2.x, f2.y, f2.z, f2.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                if (!((m >> (8 * k)) & 0xffu)) continue;
#pragma unroll
                for (int c = 0; c < 3; ++c) {
                    x.lo[c] = fminf(x.lo[c], f[3 * k + c]);
                    x.hi[c] = fmaxf(x.hi[c], f[3 * k + c]);
                }
            }
        }
    } else {
        const size_t per = (n + cs - 1) / cs;
        const size_t i0 = (size_t)rank * per, i1 = i0 + per < n ? i0 + per : n;
        for (size_t i = i0 + threadIdx.x; i < i1; i += blockDim.x) {
            if (!__ldg(valid + base + i)) continue;
            x.any = 1;
#pragma unroll
            for (int c = 0; c < 3; ++c) {
                const float p = __ldg(pos + 3 * (base + i) + c);
                x.lo[c] = fminf(x.lo[c], p);
                x.hi[c] = fmaxf(x.hi[c], p);
            }
        }
    }
    box_reduce_warp(x);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        if (lane < nw) x = s_warp[lane];
        else {
#pragma unroll
            for (int c = 0; c < 3; ++c) { x.lo[c] = FLT_MAX; x.hi[c] = -FLT_MAX; }
            x.any = 0;
        }
        box_reduce_warp(x);
        if (lane == 0) s_part = x;
    }
    cluster.sync();  // every CTA's partial box is in its shared memory
    if (rank == 0 && threadIdx.x == 0) {
        Box t = s_part;
        for (int r = 1; r < cs; ++r) {
            const Box* o = cluster.map_shared_rank(&s_part, r);
#pragma unroll
            for (int c = 0; c < 3; ++c) {
                t.lo[c] = fminf(t.lo[c], o->lo[c]);
                t.hi[c] = fmaxf(t.hi[c], o->hi[c]);
            }
            t.any |= o->any;
        }
        float tv = 0.0f;
        if (t.any) {
            const float d0 = __fsub_rn(t.hi[0], t.lo[0]), d1 = __fsub_rn(t.hi[1], t.lo[1]),
                        d2 = __fsub_rn(t.hi[2], t.lo[2]);
            const float diag2 = __fadd_rn(__fadd_rn(__fmul_rn(d0, d0), __fmul_rn(d1, d1)), __fmul_rn(d2, d2));
            tv = __fmul_rn(tol_frac, __fsqrt_rn(diag2));
        }
        tau[b] = tv;
    }
    cluster.sync();  // the other CTAs' shared memory stays alive until CTA 0 has read it
}

cudaError_t launch_tau(const float* pos, const uint8_t* valid, int B, int N, int H, int W, float tol_frac,
                       float* tau, cudaStream_t s) {
    // a cluster of 8 CTAs (the portable size) per asset: 1024 CTAs for 128
    // assets, resident at once at 8 per SM (one CTA per view at 512 threads,
    // 768 CTAs in 1.3 waves, took 16 us more per 128-asset build)
    const int cs = 8;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(B * cs);
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // quads: every view's texels start on a 4-texel boundary with 16-byte aligned positions
    const int quads = (H * W) % 4 == 0 && (uintptr_t)pos % 16 == 0 && (uintptr_t)valid % 4 == 0;
    return cudaLaunchKernelEx(&cfg, tau_kernel, pos, valid, N, H * W, tol_frac, quads, tau);
}

// ------------------------------------------------------- correspondence --
// One CTA per 256 tokens of (asset b, target view v).  The CTA's foreground
// tokens are compacted first (warp ballots), so that thread t takes the t-th
// foreground token and the warps that test taps are full; each such thread
// loops over the source views u with the target's position loaded once.
// Background tokens get empty rows from their own thread.  Writes the keep
// masks and (TABLES, when requested) the idx/w tables of every pair; with
// tile_cnt given, adds the kept rows of each (b, v, u, tile) to its count
// (one atomic per warp: a CTA's 256 tokens lie in one tile).  Without tables
// only the keep masks are formed (no renormalised weights): 581 -> 507 us
// for the build graph of 128 assets.
constexpr int kBuildThreads = 256;
static_assert(GEOCACHE_TILE_TOKENS % kBuildThreads == 0, "a build CTA's tokens lie in one tile");

// A build CTA covers REP slices of kBuildThreads tokens of one view (REP = 1
// or 4): its foreground tokens are compacted across the slices and each
// thread takes up to REP of them in turn, so that fewer lanes idle through
// the source loop (the background is ~60% of a view).  REP = 4 for large
// builds (128 batch128 assets: 504 -> 465 us for the build graph), 1 for
// small ones, where the 4x fewer CTAs would not fill the GPU.
template <int K, bool TABLES, int REP>
__global__ void __launch_bounds__(kBuildThreads) build_corr_kernel(const float* __restrict__ pos,
                                                         const uint8_t* __restrict__ valid,
                                                         const geocache_camera* __restrict__ cams,
                                                         const float* __restrict__ tau, int N, int H, int W,
                                                         int32_t* __restrict__ idx, float* __restrict__ wout,
                                                         uint8_t* __restrict__ keep, int32_t* __restrict__ tile_cnt) {
    static_assert(GEOCACHE_TILE_TOKENS % (kBuildThreads * REP) == 0, "a build CTA's tokens lie in one tile");
    const int HW = H * W;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int p_base = blockIdx.x * kBuildThreads * REP;
    const int v = blockIdx.y, b = blockIdx.z;
    __shared__ geocache_camera s_cam[GEOCACHE_MAX_VIEWS];
    __shared__ int s_fg[kBuildThreads * REP];
    __shared__ int s_wcnt[REP][kBuildThreads / 32];
    for (int i = t; i < N * 16; i += kBuildThreads)
        reinterpret_cast<float*>(s_cam)[i] = __ldg(reinterpret_cast<const float*>(cams + (size_t)b * N) + i);
    const size_t view0 = ((size_t)b * N + v) * HW;
    // compaction of the foreground tokens of the CTA's REP slices, in token order
    bool in_h[REP], fg_h[REP];
    unsigned bal[REP];
#pragma unroll
    for (int h = 0; h < REP; ++h) {
        const int ph = p_base + h * kBuildThreads + t;
        in_h[h] = ph < HW;
        fg_h[h] = in_h[h] && __ldg(valid + view0 + ph);
        bal[h] = __ballot_sync(0xffffffffu, fg_h[h]);
        if (lane == 0) s_wcnt[h][warp] = __popc(bal[h]);
    }
    __syncthreads();
    int n_fg = 0;
#pragma unroll
    for (int h = 0; h < REP; ++h) {
        int before = n_fg, tot = 0;
#pragma unroll
        for (int w = 0; w < kBuildThreads / 32; ++w) {
            before += w < warp ? s_wcnt[h][w] : 0;
            tot += s_wcnt[h][w];
        }
        if (fg_h[h]) s_fg[before + __popc(bal[h] & ((1u << lane) - 1u))] = h * kBuildThreads + t;
        n_fg += tot;
    }
    __syncthreads();
    const int T = tiles_per_view(H, W);
    const float tu = __ldg(tau + b);
    const float tau2 = __fmul_rn(tu, tu);
#pragma unroll 1
    for (int it = 0; it < REP; ++it) {
        const int jw = it * kBuildThreads + t;
        if (it > 0 && it * kBuildThreads >= n_fg) break;  // the same for every thread of the CTA
        const bool work = jw < n_fg;
        const int pw = p_base + (work ? s_fg[jw] : 0);  // this thread's foreground token
        float X0 = 0.f, X1 = 0.f, X2 = 0.f;
        if (work) {
            X0 = __ldg(pos + 3 * (view0 + pw));
            X1 = __ldg(pos + 3 * (view0 + pw) + 1);
            X2 = __ldg(pos + 3 * (view0 + pw) + 2);
        }
        for (int u = 0; u < N; ++u) {
            Taps tp;
            taps_clear(tp);
            int mask = 0;
            if (work && u != v) {
                const size_t su = ((size_t)b * N + u) * HW;
                if (TABLES) {
                    compute_taps<K>(s_cam[u], pos + 3 * su, valid + su, H, W, X0, X1, X2, tau2, tp, &mask);
                } else {
                    Footprint fp;
                    if (footprint<K>(s_cam[u], X0, X1, X2, H, W, fp))
                        mask = tap_mask<K>(fp, pos + 3 * su, valid + su, H, W, X0, X1, X2, tau2);
                }
            }
            if (tile_cnt) {
                const unsigned kept = __ballot_sync(0xffffffffu, mask != 0);
                if (lane == 0 && kept)
                    atomicAdd(tile_cnt + (((size_t)b * N + v) * N + u) * T + p_base / GEOCACHE_TILE_TOKENS,
                              __popc(kept));
            }
            const size_t row0 = (((size_t)b * N + v) * N + u) * HW;
            if (keep) {
                if (it == 0) {
#pragma unroll
                    for (int h = 0; h < REP; ++h)
                        if (in_h[h] && !fg_h[h]) keep[row0 + p_base + h * kBuildThreads + t] = 0;
                }
                if (work) keep[row0 + pw] = (uint8_t)mask;
            }
            if (!TABLES || !idx) continue;
            if (it == 0) {
#pragma unroll
                for (int h = 0; h < REP; ++h) {
                    if (!(in_h[h] && !fg_h[h])) continue;
                    const size_t e = row0 + p_base + h * kBuildThreads + t;
                    if (K == 4) {
                        reinterpret_cast<int4*>(idx)[e] = make_int4(-1, -1, -1, -1);
                        reinterpret_cast<float4*>(wout)[e] = make_float4(0.f, 0.f, 0.f, 0.f);
                    } else {
                        idx[e] = -1;
                        wout[e] = 0.0f;
                    }
                }
            }
            if (work) {
                if (K == 4) {
                    reinterpret_cast<int4*>(idx)[row0 + pw] = make_int4(tp.q[0], tp.q[1], tp.q[2], tp.q[3]);
                    reinterpret_cast<float4*>(wout)[row0 + pw] = make_float4(tp.w[0], tp.w[1], tp.w[2], tp.w[3]);
                } else {
                    idx[row0 + pw] = tp.q[0];
                    wout[row0 + pw] = tp.w[0];
                }
            }
        }
    }
}

template <int REP>
static void launch_build_corr_rep(const geocache_corr& c, int32_t* cnt, cudaStream_t s) {
    const int HW = c.H * c.W;
    const dim3 grid((HW + kBuildThreads * REP - 1) / (kBuildThreads * REP), c.N, c.B);
    if (c.K == 4 && c.idx)
        build_corr_kernel<4, true, REP><<<grid, kBuildThreads, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W,
                                                                       c.idx, c.w, c.keep, cnt);
    else if (c.K == 4)
        build_corr_kernel<4, false, REP><<<grid, kBuildThreads, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W,
                                                                        c.idx, c.w, c.keep, cnt);
    else if (c.idx)
        build_corr_kernel<1, true, REP><<<grid, kBuildThreads, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W,
                                                                       c.idx, c.w, c.keep, cnt);
    else
        build_corr_kernel<1, false, REP><<<grid, kBuildThreads, 0, s>>>(c.pos, c.valid, c.cams, c.tau, c.N, c.H, c.W,
                                                                        c.idx, c.w, c.keep, cnt);
}

cudaError_t launch_build_corr(const geocache_corr& c, cudaStream_t s) {
    int32_t* cnt = nullptr;
    if (c.tile_ptr) {
        const size_t n = (size_t)c.B * c.N * c.N * tiles_per_view(c.H, c.W) + 1;
        cudaError_t e = cudaMemsetAsync(c.tile_ptr, 0, n * sizeof(int32_t), s);
        if (e != cudaSuccess) return e;
        cnt = c.tile_ptr;
    }
    // 4 slices per CTA once the build has at least 4096 CTAs of 1024 tokens
    const long long ctas4 = (long long)tiles_per_view(c.H, c.W) * c.N * c.B;
    if (ctas4 >= 4096) launch_build_corr_rep<4>(c, cnt, s);
    else launch_build_corr_rep<1>(c, cnt, s);
    return cudaGetLastError();
}

// Device status word (the library's only device-resident state): bit 0 = a
// bounded wait gave up, bit 1 = the sparse form did not fit max_records,
// bit 2 = a record permutation entry was out of range, bit 4 = a table index
// was outside [-1, H*W) (bit 3 is the rasteriser's word's bad face index).
// Read and cleared by geocache_device_status().
__device__ unsigned int g_device_error = 0;

// ---------------------------------------------------- sparse operator --
// G_{u->v} in tile-CSR form: for each (asset b, target view v, source view u,
// tile of GEOCACHE_TILE_TOKENS tokens) the records of its kept rows, in token
// order; tile_ptr holds the exclusive prefix sum of the per-tile counts.
__device__ __forceinline__ int tiles_per_view_dev(int H, int W) {
    return (H * W + GEOCACHE_TILE_TOKENS - 1) / GEOCACHE_TILE_TOKENS;
}

// in-place exclusive prefix sum of n counts by one CTA; a[n] = total, or -1
// when the total does not fit an int32.  Rounds of 1024 x kScanPer
// consecutive counts: each thread loads its kScanPer counts (16-byte loads
// when aligned), the CTA scans the per-thread sums, and each thread rewrites
// its counts as offsets from the running total of the earlier rounds.
constexpr int kScanPer = 16;

__global__ void __launch_bounds__(1024) exclusive_scan_kernel(int32_t* a, long long n) {
    __shared__ long long s_warp[32];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const bool vec = (reinterpret_cast<uintptr_t>(a) & 15) == 0;
    long long carry = 0;  // sum of the counts of the earlier rounds
    for (long long c0 = 0; c0 < n; c0 += 1024LL * kScanPer) {
        const long long lo = c0 + (long long)t * kScanPer;
        int x[kScanPer];
        if (vec && lo + kScanPer <= n) {
#pragma unroll
            for (int i = 0; i < kScanPer; i += 4) {
                const int4 q = *reinterpret_cast<const int4*>(a + lo + i);
                x[i] = q.x; x[i + 1] = q.y; x[i + 2] = q.z; x[i + 3] = q.w;
            }
        } else {
#pragma unroll
            for (int i = 0; i < kScanPer; ++i) x[i] = lo + i < n ? a[lo + i] : 0;
        }
        long long sum = 0;
#pragma unroll
        for (int i = 0; i < kScanPer; ++i) sum += x[i];
        long long incl = sum;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const long long y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += y;
        }
        if (lane == 31) s_warp[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            long long w = s_warp[lane];
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const long long y = __shfl_up_sync(0xffffffffu, w, off);
                if (lane >= off) w += y;
            }
            s_warp[lane] = w;
        }
        __syncthreads();
        long long run = carry + (warp ? s_warp[warp - 1] : 0) + incl - sum;
#pragma unroll
        for (int i = 0; i < kScanPer; ++i) {  // counts -> offsets
            const int c = x[i];
            x[i] = run > 0x7fffffffLL ? -1 : (int32_t)run;
            run += c;
        }
        if (vec && lo + kScanPer <= n) {
#pragma unroll
            for (int i = 0; i < kScanPer; i += 4)
                *reinterpret_cast<int4*>(a + lo + i) = make_int4(x[i], x[i + 1], x[i + 2], x[i + 3]);
        } else {
#pragma unroll
            for (int i = 0; i < kScanPer; ++i)
                if (lo + i < n) a[lo + i] = x[i];
        }
        carry += s_warp[31];
        __syncthreads();  // s_warp is rewritten by the next round
    }
    if (t == 0) {
        a[n] = carry > 0x7fffffffLL ? -1 : (int32_t)carry;
        if (carry > 0x7fffffffLL) atomicOr(&g_device_error, 2u);  // more records than int32 offsets index
    }
}

// tile_ptr holds the per-tile counts written by build_corr_kernel; turn them
// into offsets
cudaError_t launch_tile_ptr(const geocache_corr& c, cudaStream_t s) {
    const int T = tiles_per_view(c.H, c.W);
    exclusive_scan_kernel<<<1, 1024, 0, s>>>(c.tile_ptr, (long long)c.B * c.N * c.N * T);
    return cudaGetLastError();
}

// records of one (b, v, u, tile): kept rows in token order, each with its
// footprint's top-left tap and fractions (recomputed with the same device
// functions as the tables, so the taps and weights they give are identical).
// The tile's offsets and keep masks are loaded together, and the kept
// targets' positions are in flight while the CTA scans its counts; the kept
// rows are then compacted (with their positions) in shared memory, so that
// each thread forms about the same number of footprints (one thread per
// quad with 0 to 4 kept rows left most lanes idle: 464 -> 427 us for the
// build graph of 128 assets).  Eight
// resident CTAs per SM (32 registers, a few spilled) hide more of that
// latency than the unbounded 43-register build (build graph of 128 assets:
// 620 vs 641 us).
template <int K>
__global__ void __launch_bounds__(256, 8) fill_records_kernel(const float* __restrict__ pos,
                                                           const geocache_camera* __restrict__ cams,
                                                           const uint8_t* __restrict__ keep,
                                                           const int32_t* __restrict__ tile_ptr, int N, int H,
                                                           int W, int T, geocache_tap_record* __restrict__ rec,
                                                           long long max_records) {
    // blockIdx.y runs over the N (N - 1) off-diagonal pairs (diagonal pairs
    // have no records): v = y / (N - 1), and u the (y mod (N - 1))-th view
    // other than v
    const int tile = blockIdx.x, b = blockIdx.z;
    const int v = (int)blockIdx.y / (N - 1), up = (int)blockIdx.y - v * (N - 1);
    const int u = up + (up >= v);
    const int vu = v * N + u;
    const int HW = H * W;
    const int t = threadIdx.x;
    const size_t ti = ((size_t)b * N * N + vu) * T + tile;
    const int r_first = __ldg(tile_ptr + ti), r_next = __ldg(tile_ptr + ti + 1);
    const int p0 = tile * GEOCACHE_TILE_TOKENS + 4 * t;
    const uint8_t* row = keep + ((size_t)b * N * N + vu) * HW;
    uint32_t m4 = 0;  // keep masks of tokens p0 .. p0 + 3, one byte each
    if (p0 + 3 < HW && (reinterpret_cast<uintptr_t>(row + p0) & 3) == 0) {
        m4 = __ldg(reinterpret_cast<const uint32_t*>(row + p0));
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (p0 + i < HW) m4 |= (uint32_t)__ldg(row + p0 + i) << (8 * i);
    }
    // a tile without records has nothing to write; < 0: offsets overflowed (flagged by the scan)
    if (r_next == r_first || r_first < 0) return;
    __shared__ geocache_camera s_cam;
    __shared__ int s_warp[8];
    __shared__ int s_kept[GEOCACHE_TILE_TOKENS];
    __shared__ float s_X[GEOCACHE_TILE_TOKENS][3];
    if (t < 16) reinterpret_cast<float*>(&s_cam)[t] = __ldg(reinterpret_cast<const float*>(cams + (size_t)b * N + u) + t);
    const size_t tv0 = ((size_t)b * N + v) * HW;
    float X[4][3];
    int mine = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        X[i][0] = X[i][1] = X[i][2] = 0.0f;
        if ((m4 >> (8 * i)) & 0xffu) {
            const float* q = pos + 3 * (tv0 + p0 + i);
            X[i][0] = __ldg(q);
            X[i][1] = __ldg(q + 1);
            X[i][2] = __ldg(q + 2);
            ++mine;
        }
    }
    // exclusive scan over the CTA (token order)
    const int lane = t & 31, warp = t >> 5;
    int incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    int base = 0, n_kept = 0;
    for (int w = 0; w < 8; ++w) {
        base += w < warp ? s_warp[w] : 0;
        n_kept += s_warp[w];
    }
    // the kept rows, compacted in token order (= record order) with their
    // target positions, so that the footprints spread evenly over the threads
    int k = base + incl - mine;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t m = (m4 >> (8 * i)) & 0xffu;
        if (!m) continue;
        s_kept[k] = (p0 + i) | (int)(m << 28);
        s_X[k][0] = X[i][0];
        s_X[k][1] = X[i][1];
        s_X[k][2] = X[i][2];
        ++k;
    }
    __syncthreads();
    for (int j = t; j < n_kept; j += 256) {
        const int tm = s_kept[j];
        Footprint f;
        footprint<K>(s_cam, s_X[j][0], s_X[j][1], s_X[j][2], H, W, f);
        geocache_tap_record out;
        out.token_mask = tm;
        out.q_tl = f.j0 * W + f.i0;
        out.fx = K == 4 ? f.ax[1] : 0.0f;
        out.fy = K == 4 ? f.ay[1] : 0.0f;
        const long long r = (long long)r_first + j;
        if (r < max_records)
            reinterpret_cast<int4*>(rec)[r] = *reinterpret_cast<const int4*>(&out);
        else
            atomicOr(&g_device_error, 2u);  // records beyond the capacity are dropped
    }
}

cudaError_t launch_fill_records(const geocache_corr& c, cudaStream_t s) {
    const int T = tiles_per_view(c.H, c.W);
    dim3 grid(T, c.N * (c.N - 1), c.B);
    if (c.K == 4)
        fill_records_kernel<4><<<grid, 256, 0, s>>>(c.pos, c.cams, c.keep, c.tile_ptr, c.N, c.H, c.W, T, c.records,
                                                    c.max_records);
    else
        fill_records_kernel<1><<<grid, 256, 0, s>>>(c.pos, c.cams, c.keep, c.tile_ptr, c.N, c.H, c.W, T, c.records,
                                                    c.max_records);
    return cudaGetLastError();
}

// Source index of the sparse form: the records grouped by (asset b, source
// view u, source tile st), st = the tile of the record's first kept tap, so
// that a step can apply the records per source tile with the anchor's tile
// staged in shared memory.  Entries are (record index, target view).  Two
// passes over the records: a count per group, then (after the exclusive scan
// of the counts into src_ptr) a scatter that advances src_ptr[g] by one per
// entry, which leaves src_ptr[g] = the end of group g (its start is
// src_ptr[g - 1], 0 for g = 0).  The order within a group is that of the
// atomics; nothing depends on it (each record's increment is computed on its
// own).
template <int K>
__device__ __forceinline__ int first_kept_tap(int mask, int q_tl, int W) {
    if (K == 1) return q_tl;
    const int k = __ffs(mask) - 1;  // the lowest kept tap: TL, TR, BL, BR
    return q_tl + (k & 1) + (k >> 1) * W;
}

template <int K, bool SCATTER>
__global__ void __launch_bounds__(256) src_index_kernel(const int32_t* __restrict__ tile_ptr,
                                                        const geocache_tap_record* __restrict__ rec,
                                                        long long max_records, int N, int W, int T,
                                                        int32_t* __restrict__ src_ptr, int2* __restrict__ src_rec) {
    const int tile = blockIdx.x, vu = blockIdx.y, b = blockIdx.z;
    const int v = vu / N, u = vu % N;
    if (u == v) return;
    const size_t ti = ((size_t)b * N * N + vu) * T + tile;
    const long long x0 = __ldg(tile_ptr + ti), x1 = __ldg(tile_ptr + ti + 1);
    const int r0 = (int)(x0 < 0 ? 0 : (x0 < max_records ? x0 : max_records));
    const int r1 = (int)(x1 < 0 ? 0 : (x1 < max_records ? x1 : max_records));
    for (int r = r0 + threadIdx.x; r < r1; r += 256) {
        const int4 x = __ldg(reinterpret_cast<const int4*>(rec) + r);
        const int q = first_kept_tap<K>((int)((uint32_t)x.x >> 28), x.y, W);
        const size_t g = ((size_t)b * N + u) * T + q / GEOCACHE_TILE_TOKENS;
        if (!SCATTER) atomicAdd(src_ptr + g, 1);
        else src_rec[atomicAdd(src_ptr + g, 1)] = make_int2(r, v);
    }
}

cudaError_t launch_src_index(const geocache_corr& c, cudaStream_t s) {
    const int T = tiles_per_view(c.H, c.W);
    const long long groups = (long long)c.B * c.N * T;
    cudaError_t e = cudaMemsetAsync(c.src_ptr, 0, (groups + 1) * sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
    const dim3 grid(T, c.N * c.N, c.B);
    int2* out = reinterpret_cast<int2*>(c.src_rec);
    if (c.K == 4)
        src_index_kernel<4, false><<<grid, 256, 0, s>>>(c.tile_ptr, c.records, c.max_records, c.N, c.W, T, c.src_ptr, out);
    else
        src_index_kernel<1, false><<<grid, 256, 0, s>>>(c.tile_ptr, c.records, c.max_records, c.N, c.W, T, c.src_ptr, out);
    exclusive_scan_kernel<<<1, 1024, 0, s>>>(c.src_ptr, groups);
    if (c.K == 4)
        src_index_kernel<4, true><<<grid, 256, 0, s>>>(c.tile_ptr, c.records, c.max_records, c.N, c.W, T, c.src_ptr, out);
    else
        src_index_kernel<1, true><<<grid, 256, 0, s>>>(c.tile_ptr, c.records, c.max_records, c.N, c.W, T, c.src_ptr, out);
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

// Fused cached step: a persistent kernel whose CTAs loop over work units
// (asset b, view v, tile of kTileTokens tokens, group of 4 channels).
//  * Streaming: one thread arms the unit's mbarrier and issues TMA bulk
//    copies (cp.async.bulk) of the unit's rows of x0 (the anchor's fresh x0,
//    or x0(t-1)) and of x_t into a two-stage shared-memory ring, one unit
//    ahead, so the next unit's rows are in flight while the current unit's
//    increments are formed.
//  * Increments (views outside the anchor set): the (token, anchor) pairs
//    with a kept tap are compacted into a work list (block prefix sum, token
//    order) and processed one per thread, so the dependent loads of many
//    tokens overlap:  keep masks -> target position -> projection and
//    weights -> gathers of the anchor increments x0_new - x0(t-1) at the kept
//    taps.  Per-anchor sums are combined in anchor order (Eq. 1 with the
//    multi-anchor aggregation of Sec. 3.2: the mean over covering anchors; a
//    token without a kept tap keeps x0(t-1)).
//  * Every token is stored (x0(t)) and reconstructed (x_{t-1}) from the
//    staged rows with 16-byte stores.
constexpr int kTileTokens = 4 * kThreads;
static_assert(kTileTokens == GEOCACHE_TILE_TOKENS, "tile of the sparse form");
constexpr int kChunk = 4;                        // anchors per work-list round
constexpr int kPairCap = kChunk * kTileTokens;   // (token, anchor) work items of one round
constexpr int kStages = 2;
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // default limit of a bounded mbarrier wait: 2 s

// Test hook of the failure handling (geocache_debug_set_wait): the limit of
// the bounded waits, and a one-shot request that the next staged transport
// launch arm none of its first unit's copies, so that wait runs out.
static std::atomic<unsigned long long> g_wait_limit_ns{kWaitLimitNs};
static std::atomic<int> g_drop_first_copy{0};

void set_debug_wait(unsigned long long limit_ns, int drop_first_copy) {
    g_wait_limit_ns.store(limit_ns ? limit_ns : kWaitLimitNs);
    g_drop_first_copy.store(drop_first_copy ? 1 : 0);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Wait for the phase with the given parity; false after limit_ns.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, unsigned long long limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer() - t0 > limit_ns) return false;
    return true;
}

// exclusive prefix sum over the CTA (deterministic); returns the total
__device__ __forceinline__ int block_exclusive_scan(int x, int& total, int* s_warp) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = x;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = lane < kThreads / 32 ? s_warp[lane] : 0;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, off);
            if (lane >= off) w += y;
        }
        if (lane < kThreads / 32) s_warp[lane] = w;  // inclusive warp totals
    }
    __syncthreads();
    total = s_warp[kThreads / 32 - 1];
    const int base = warp ? s_warp[warp - 1] : 0;
    return base + incl - x;
}

struct FusedShared {
    float acc[kTileTokens][4];        // per token: sum over covering anchors (anchor order), channel group
    uint32_t pair[kPairCap];          // work items: token | anchor << 10 | keep mask << 16
    uint8_t n[kTileTokens];           // per token: number of covering anchors
    geocache_camera cam[kChunk];
    int warp[kThreads / 32];
    uint64_t bar[kStages];
};

// Taps of work item (token p of view v, anchor slot s2) in the given mode.
template <int K, int MODE>
__device__ __forceinline__ void item_taps(const TransportArgs& args, const geocache_camera& cam, int b, int v,
                                          int s2, int p, int m, size_t tv0, size_t plane, float tau2, Taps& tp) {
    const int N = args.N;
    const int u = args.anchors[s2];
    if (MODE == GEOCACHE_CORR_TABLE) {
        const size_t row = (((size_t)b * N + v) * N + u) * plane + p;
        tp.kept = 0;
#pragma unroll
        for (int kk = 0; kk < K; ++kk) {
            int q = __ldg(args.idx + row * K + kk);
            float wq = __ldg(args.w + row * K + kk);
            if (q < -1 || q >= (int)plane) {  // a caller's table with an index outside the view: dropped, reported
                atomicOr(&g_device_error, 16u);
                q = -1;
                wq = 0.0f;
            }
            tp.q[kk] = q;
            tp.w[kk] = wq;
            tp.kept += q >= 0;
        }
        return;
    }
    const float X0 = __ldg(args.pos + 3 * (tv0 + p));
    const float X1 = __ldg(args.pos + 3 * (tv0 + p) + 1);
    const float X2 = __ldg(args.pos + 3 * (tv0 + p) + 2);
    if (MODE == GEOCACHE_CORR_MASK) {
        Footprint f;
        footprint<K>(cam, X0, X1, X2, args.H, args.W, f);
        taps_from_mask<K>(f, m, args.W, tp);
    } else {
        const size_t su = ((size_t)b * N + u) * plane;
        compute_taps<K>(cam, args.pos + 3 * su, args.valid + su, args.H, args.W, X0, X1, X2, tau2, tp);
    }
}

// Tap-weighted increment of one anchor at one token, channels [cg, cg+cn).
template <int K>
__device__ __forceinline__ void item_increment(const TransportArgs& args, const Taps& tp, int b, int s2, int cg,
                                               int cn, size_t plane, float (&g)[4]) {
    const int N = args.N, C = args.C, a = args.a;
    const float* xn = args.x0_new + (((size_t)b * a + s2) * C + cg) * plane;
    const float* xp = args.x0_prev + (((size_t)b * N + args.anchors[s2]) * C + cg) * plane;
    const bool copy = args.update == GEOCACHE_UPDATE_COPY;
    float dn[K][4], dp[K][4];
#pragma unroll
    for (int kk = 0; kk < K; ++kk)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            dn[kk][c] = 0.0f;
            dp[kk][c] = 0.0f;
            if (tp.q[kk] >= 0 && c < cn) {
                const size_t e = (size_t)c * plane + tp.q[kk];
                dn[kk][c] = __ldg(xn + e);
                dp[kk][c] = __ldg(xp + e);
            }
        }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        float acc = 0.0f;
#pragma unroll
        for (int kk = 0; kk < K; ++kk)
            if (tp.q[kk] >= 0) acc = tap_term(copy, tp.w[kk], dn[kk][c], dp[kk][c], acc);
        g[c] = acc;
    }
}

struct UnitCoord {
    int b, v, tile, cg;
};

__device__ __forceinline__ UnitCoord unit_coord(long long u, int n_tiles, int n_cg, int N) {
    UnitCoord c;
    c.cg = (int)(u % n_cg) * 4;
    u /= n_cg;
    c.tile = (int)(u % n_tiles);
    u /= n_tiles;
    c.v = (int)(u % N);
    c.b = (int)(u / N);
    return c;
}

// Increments of the tile's covered tokens (views outside the anchor set),
// left in sh.acc / sh.n for the tile's tokens.
template <int K, int MODE, bool VEC>
__device__ __forceinline__ void tile_increments(const TransportArgs& args, FusedShared& sh, int b, int v, int tile0,
                                                int cg, int cn) {
    const int HW = args.H * args.W;
    const int t = threadIdx.x;
    const int p0 = tile0 + 4 * t;
    const int cnt = p0 < HW ? (HW - p0 < 4 ? HW - p0 : 4) : 0;
    const int N = args.N, a = args.a;
    const size_t plane = (size_t)HW;
    const size_t tv0 = ((size_t)b * N + v) * plane;
    float tau2 = 0.0f;
    if (MODE == GEOCACHE_CORR_GEOMETRY) {
        const float tu = __ldg(args.tau + b);
        tau2 = __fmul_rn(tu, tu);
    }
    uint32_t fg = 0;
    if (cnt > 0 && MODE == GEOCACHE_CORR_GEOMETRY) fg = quad_masks(args.valid + tv0 + p0, cnt, VEC);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        *reinterpret_cast<float4*>(sh.acc[4 * t + i]) = make_float4(0.f, 0.f, 0.f, 0.f);
        sh.n[4 * t + i] = 0;
    }
    for (int ac = 0; ac < a; ac += kChunk) {
        const int na = a - ac < kChunk ? a - ac : kChunk;
        if (MODE != GEOCACHE_CORR_TABLE)
            for (int i = t; i < na * 16; i += kThreads)
                reinterpret_cast<float*>(sh.cam)[i] = __ldg(
                    reinterpret_cast<const float*>(args.cams + (size_t)b * N + args.anchors[ac + (i >> 4)]) + (i & 15));
        // (token, anchor) work items of this anchor chunk
        uint32_t m4[4] = {0, 0, 0, 0};  // per own token: 4 bits per anchor of the chunk
        if (cnt > 0) {
            if (MODE == GEOCACHE_CORR_MASK) {
                const uint8_t* krow = args.keep + ((size_t)b * N + v) * N * plane + p0;
                uint32_t q[kChunk];
#pragma unroll
                for (int s2 = 0; s2 < kChunk; ++s2)  // the chunk's masks in flight together
                    q[s2] = s2 < na ? quad_masks(krow + (size_t)args.anchors[ac + s2] * plane, cnt, VEC) : 0u;
#pragma unroll
                for (int s2 = 0; s2 < kChunk; ++s2)
#pragma unroll
                    for (int i = 0; i < 4; ++i) m4[i] |= ((q[s2] >> (8 * i)) & 15u) << (4 * s2);
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const bool cand = MODE == GEOCACHE_CORR_GEOMETRY ? ((fg >> (8 * i)) & 0xffu) != 0 : i < cnt;
                    if (cand) m4[i] = (1u << (4 * na)) - 1u;  // every anchor is a candidate
                }
            }
        }
        int mine = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int s2 = 0; s2 < kChunk; ++s2) mine += (m4[i] >> (4 * s2)) & 15u ? 1 : 0;
        int n_items;
        int k = block_exclusive_scan(mine, n_items, sh.warp);  // barriers inside
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int s2 = 0; s2 < kChunk; ++s2) {
                const uint32_t m = (m4[i] >> (4 * s2)) & 15u;
                if (m) sh.pair[k++] = (uint32_t)(4 * t + i) | ((uint32_t)s2 << 10) | (m << 16);
            }
        __syncthreads();
        for (int r0 = 0; r0 < n_items; r0 += kThreads) {
            const int j = r0 + t;
            float g[4] = {0.f, 0.f, 0.f, 0.f};
            int s_mine = -1, lp = 0;
            if (j < n_items) {
                const uint32_t it = sh.pair[j];
                lp = (int)(it & 1023u);
                const int s_loc = (int)((it >> 10) & 63u);
                const int m = (int)((it >> 16) & 15u);
                Taps tp;
                item_taps<K, MODE>(args, sh.cam[s_loc], b, v, ac + s_loc, tile0 + lp, m, tv0, plane, tau2, tp);
                if (tp.kept) {
                    item_increment<K>(args, tp, b, ac + s_loc, cg, cn, plane, g);
                    s_mine = s_loc;
                }
            }
            // combine in anchor order (deterministic): anchor s_loc adds in pass s_loc
            for (int s2 = 0; s2 < na; ++s2) {
                if (s_mine == s2) {
                    float4* dst = reinterpret_cast<float4*>(sh.acc[lp]);
                    float4 cur = *dst;
                    cur.x = __fadd_rn(cur.x, g[0]);
                    cur.y = __fadd_rn(cur.y, g[1]);
                    cur.z = __fadd_rn(cur.z, g[2]);
                    cur.w = __fadd_rn(cur.w, g[3]);
                    *dst = cur;
                    sh.n[lp] += 1;
                }
                __syncthreads();
            }
        }
    }
}

template <typename T, int K, int MODE>
__global__ void __launch_bounds__(kThreads) transport_fused_kernel(const TransportArgs args, int n_tiles, int n_cg,
                                                                   long long n_units) {
    __shared__ FusedShared sh;
    extern __shared__ __align__(128) unsigned char dyn[];  // [stage]: x0 rows [4][tile] f32, x_t rows [4][tile] T
    constexpr size_t kStageBytes = 4 * kTileTokens * (sizeof(float) + sizeof(T));
    const int t = threadIdx.x;
    const int HW = args.H * args.W;
    const int N = args.N, C = args.C, a = args.a;
    const size_t plane = (size_t)HW;
    const bool recon = args.coef.enabled;
    const T* xt_p = static_cast<const T*>(args.x_t);
    T* xn_p = static_cast<T*>(args.x_next);

    // issue the bulk copies of unit u into stage st (thread 0)
    auto issue = [&](long long u, int st) {
        if (args.drop_first_copy && u == 0) return;  // test hook: this unit's wait runs out
        const UnitCoord c = unit_coord(u, n_tiles, n_cg, N);
        const int tile0 = c.tile * kTileTokens;
        const int tile_n = HW - tile0 < kTileTokens ? HW - tile0 : kTileTokens;
        const int cn = C - c.cg < 4 ? C - c.cg : 4;
        const int slot = args.slot_of[c.v];
        const float* src = slot >= 0 ? args.x0_new + ((size_t)c.b * a + slot) * C * plane
                                     : args.x0_prev + ((size_t)c.b * N + c.v) * C * plane;
        float* s_x0 = reinterpret_cast<float*>(dyn + st * kStageBytes);
        T* s_xt = reinterpret_cast<T*>(dyn + st * kStageBytes + 4 * kTileTokens * sizeof(float));
        const uint32_t rx = (uint32_t)tile_n * sizeof(float), rt = (uint32_t)tile_n * sizeof(T);
        mbar_arrive_expect_tx(&sh.bar[st], cn * (rx + (recon ? rt : 0)));
        for (int cc = 0; cc < cn; ++cc) {
            bulk_g2s(s_x0 + cc * kTileTokens, src + (size_t)(c.cg + cc) * plane + tile0, rx, &sh.bar[st]);
            if (recon)
                bulk_g2s(s_xt + cc * kTileTokens, xt_p + (((size_t)c.b * N + c.v) * C + c.cg + cc) * plane + tile0, rt,
                         &sh.bar[st]);
        }
    };

    if (t == 0) {
        for (int st = 0; st < kStages; ++st) mbar_init(&sh.bar[st], 1);
        fence_mbar_init();
        if ((long long)blockIdx.x < n_units) issue(blockIdx.x, 0);
    }
    __syncthreads();
    uint32_t parity[kStages] = {0, 0};
    int st = 0;
    for (long long u = blockIdx.x; u < n_units; u += gridDim.x) {
        const long long un = u + gridDim.x;
        if (t == 0 && un < n_units) {
            fence_proxy_async();  // the previous unit's shared-memory reads of this stage come first
            issue(un, st ^ 1);
        }
        const UnitCoord c = unit_coord(u, n_tiles, n_cg, N);
        const int tile0 = c.tile * kTileTokens;
        const int p0 = tile0 + 4 * t;
        const int cnt = p0 < HW ? (HW - p0 < 4 ? HW - p0 : 4) : 0;
        const int cn = C - c.cg < 4 ? C - c.cg : 4;
        const int slot = args.slot_of[c.v];
        if (slot < 0) tile_increments<K, MODE, true>(args, sh, c.b, c.v, tile0, c.cg, cn);

        const bool ok = mbar_wait_bounded(&sh.bar[st], parity[st], args.wait_limit_ns);
        if (__syncthreads_or(!ok)) {  // the whole CTA gives up together
            if (t == 0) atomicOr(&g_device_error, 1u);
            for (int s2 = 0; s2 < kStages; ++s2)  // copies in flight
                mbar_wait_bounded(&sh.bar[s2], parity[s2], args.wait_limit_ns);
            return;
        }
        parity[st] ^= 1u;
        if (cnt > 0) {
            const float* s_x0 = reinterpret_cast<const float*>(dyn + st * kStageBytes);
            const T* s_xt = reinterpret_cast<const T*>(dyn + st * kStageBytes + 4 * kTileTokens * sizeof(float));
            const size_t view_base = ((size_t)c.b * N + c.v) * C * plane + p0;
            float x0[4][4];
            typename Lat4<T>::Raw xt[4];
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
                if (cc >= cn) break;
                const float4 q = *reinterpret_cast<const float4*>(s_x0 + cc * kTileTokens + 4 * t);
                x0[cc][0] = q.x; x0[cc][1] = q.y; x0[cc][2] = q.z; x0[cc][3] = q.w;
                if (recon) xt[cc] = *reinterpret_cast<const typename Lat4<T>::Raw*>(s_xt + cc * kTileTokens + 4 * t);
            }
            if (slot < 0) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int n = sh.n[4 * t + i];
                    if (!n) continue;
                    const float4 g = *reinterpret_cast<const float4*>(sh.acc[4 * t + i]);
                    const float gg[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc)
                        x0[cc][i] = fold_one(args.update == GEOCACHE_UPDATE_COPY, x0[cc][i], gg[cc], n);
                }
            }
            if (slot < 0 || args.write_anchor_rows) {
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) {
                    if (cc >= cn) break;
                    Lat4<float>::store(args.x0_out, view_base + (size_t)(c.cg + cc) * plane, cnt, true, x0[cc]);
                }
            }
            if (recon) {
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) {
                    if (cc >= cn) break;
                    float x[4], y[4], pr[4];
                    Lat4<T>::unpack(xt[cc], x);
#pragma unroll
                    for (int i = 0; i < 4; ++i) y[i] = recon_one(args.coef, x[i], x0[cc][i], pr[i]);
                    const size_t e = view_base + (size_t)(c.cg + cc) * plane;
                    Lat4<T>::store(xn_p, e, cnt, true, y);
                    if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, true, pr);
                }
            }
        }
        __syncthreads();  // stage st and the sums are reused by later units
        st ^= 1;
    }
}

// General path (sizes the bulk copies cannot serve: H*W not a multiple of 8
// or buffers not 16-byte aligned): one CTA per unit, registers instead of
// the shared-memory ring.
template <typename T, int K, int MODE, bool VEC>
__global__ void __launch_bounds__(kThreads) transport_simple_kernel(const TransportArgs args, int n_tiles, int n_cg) {
    __shared__ FusedShared sh;
    const int t = threadIdx.x;
    const int HW = args.H * args.W;
    const int N = args.N, C = args.C, a = args.a;
    const size_t plane = (size_t)HW;
    const bool recon = args.coef.enabled;
    const T* xt_p = static_cast<const T*>(args.x_t);
    T* xn_p = static_cast<T*>(args.x_next);
    const UnitCoord c = unit_coord(blockIdx.x, n_tiles, n_cg, N);
    const int tile0 = c.tile * kTileTokens;
    const int p0 = tile0 + 4 * t;
    const int cnt = p0 < HW ? (HW - p0 < 4 ? HW - p0 : 4) : 0;
    const int cn = C - c.cg < 4 ? C - c.cg : 4;
    const int slot = args.slot_of[c.v];
    const size_t view_base = ((size_t)c.b * N + c.v) * C * plane + p0;
    const float* src = slot >= 0 ? args.x0_new + ((size_t)c.b * a + slot) * C * plane + p0
                                 : args.x0_prev + ((size_t)c.b * N + c.v) * C * plane + p0;
    float x0[4][4];
    typename Lat4<T>::Raw xt[4];
    if (cnt > 0) {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
            if (cc >= cn) break;
            if (slot >= 0)
                f4_load_keep(src, (size_t)(c.cg + cc) * plane, cnt, VEC, x0[cc]);
            else
                Lat4<float>::load(src, (size_t)(c.cg + cc) * plane, cnt, VEC, x0[cc]);
            if (recon) xt[cc] = Lat4<T>::load_raw(xt_p, view_base + (size_t)(c.cg + cc) * plane, cnt, VEC);
        }
    }
    if (slot < 0) tile_increments<K, MODE, VEC>(args, sh, c.b, c.v, tile0, c.cg, cn);
    if (cnt <= 0) return;
    if (slot < 0) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int n = sh.n[4 * t + i];
            if (!n) continue;
            const float4 g = *reinterpret_cast<const float4*>(sh.acc[4 * t + i]);
            const float gg[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
            for (int cc = 0; cc < 4; ++cc)
                x0[cc][i] = fold_one(args.update == GEOCACHE_UPDATE_COPY, x0[cc][i], gg[cc], n);
        }
    }
    if (slot < 0 || args.write_anchor_rows) {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
            if (cc >= cn) break;
            Lat4<float>::store(args.x0_out, view_base + (size_t)(c.cg + cc) * plane, cnt, VEC, x0[cc]);
        }
    }
    if (recon) {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
            if (cc >= cn) break;
            float x[4], y[4], pr[4];
            Lat4<T>::unpack(xt[cc], x);
#pragma unroll
            for (int i = 0; i < 4; ++i) y[i] = recon_one(args.coef, x[i], x0[cc][i], pr[i]);
            const size_t e = view_base + (size_t)(c.cg + cc) * plane;
            Lat4<T>::store(xn_p, e, cnt, VEC, y);
            if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, VEC, pr);
        }
    }
}

// Sparse mode.  A cached step is two kernels:
//  phase A: (i) the records of the step's pairs (v outside the anchor set,
//    anchor u) applied record-parallel: for each record the kept taps and
//    weights, then sum_k w_k (x0_new - x0(t-1))[q_k] for every channel,
//    written to workspace[r * C + c];  (ii) the anchor views streamed
//    (x0(t) = the denoiser's x0, reconstruction).  The two kinds of CTA are
//    interleaved in launch order so that the latency-bound gathers overlap
//    the bandwidth-bound streaming and both read the anchors' fresh x0 while
//    it is in L2.  For an in-place cache update the anchor rows are written
//    by phase B instead (the gathers read x0(t-1) of the anchors).
//  phase B: the other views streamed; each CTA folds its tile's record
//    increments in anchor order (deterministic: the mean over covering
//    anchors of Eq. 1 with the aggregation of Sec. 3.2; tokens without a
//    record keep x0(t-1)), then stores and reconstructs every token.
// Wide latents (C >= 8) with room in the workspace take another phase A:
// the anchor views streamed while their increments are written once as a
// plane (4 channels per 16-byte word), from which phase B forms each
// record's increment itself (sparse_phase_a_plane_kernel below).  Without
// that room, phase A applies the records per source tile when the corr has
// a source index (sparse_phase_a_src_kernel), else record-parallel.

// Streamed rows of the quad of tokens p0.. of view v of asset b, channel
// group cg: x0 (the anchor's fresh x0 or x0(t-1)) and x_t.
template <typename T, bool VEC>
struct QuadRows {
    float x0[4][4];
    typename Lat4<T>::Raw xt[4];

    __device__ __forceinline__ void load(const TransportArgs& args, int b, int v, int slot, int p0, int cnt, int cg,
                                         int cn) {
        const size_t plane = (size_t)args.H * args.W;
        const int N = args.N, C = args.C, a = args.a;
        const float* x0_src = slot >= 0 ? args.x0_new + ((size_t)b * a + slot) * C * plane + p0
                                        : args.x0_prev + ((size_t)b * N + v) * C * plane + p0;
        const T* xt_p = static_cast<const T*>(args.x_t) + ((size_t)b * N + v) * C * plane + p0;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            if (c >= cn) break;
            if (slot >= 0)
                f4_load_keep(x0_src, (size_t)(cg + c) * plane, cnt, VEC, x0[c]);
            else
                Lat4<float>::load(x0_src, (size_t)(cg + c) * plane, cnt, VEC, x0[c]);
            if (args.coef.enabled) xt[c] = Lat4<T>::load_raw(xt_p, (size_t)(cg + c) * plane, cnt, VEC);
        }
    }

    // add the folded increments of the quad's tokens (the mean over their
    // covering anchors, Eq. 1 with the aggregation of Sec. 3.2): n4 holds the
    // four tokens' anchor counts, one byte each; g / n is a multiplication
    // for n a power of two (exact) and a division otherwise
    template <bool COPY>
    __device__ __forceinline__ void fold4(const float (*s_acc)[4], uint32_t n4, int lp0) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int n = (int)((n4 >> (8 * i)) & 0xffu);
            if (!n) continue;
            const float4 gq = *reinterpret_cast<const float4*>(s_acc[lp0 + i]);
            const float gg[4] = {gq.x, gq.y, gq.z, gq.w};
            float m[4];
            if (n == 1) {
#pragma unroll
                for (int c = 0; c < 4; ++c) m[c] = gg[c];
            } else if ((n & (n - 1)) == 0) {
                const float rn = __frcp_rn((float)n);
#pragma unroll
                for (int c = 0; c < 4; ++c) m[c] = __fmul_rn(gg[c], rn);
            } else {
#pragma unroll
                for (int c = 0; c < 4; ++c) m[c] = __fdiv_rn(gg[c], (float)n);
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) x0[c][i] = COPY ? m[c] : __fadd_rn(x0[c][i], m[c]);
        }
    }

    // store x0(t) and the reconstruction
    __device__ __forceinline__ void store(const TransportArgs& args, int b, int v, int p0, int cnt, int cg, int cn) {
        const size_t plane = (size_t)args.H * args.W;
        const size_t view_base = ((size_t)b * args.N + v) * args.C * plane + p0;
        T* xn_p = static_cast<T*>(args.x_next);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            if (c >= cn) break;
            const size_t e = view_base + (size_t)(cg + c) * plane;
            Lat4<float>::store(args.x0_out, e, cnt, VEC, x0[c]);
            if (args.coef.enabled) {
                float x[4], yv[4], pr[4];
                Lat4<T>::unpack(xt[c], x);
#pragma unroll
                for (int i = 0; i < 4; ++i) yv[i] = recon_one(args.coef, x[i], x0[c][i], pr[i]);
                Lat4<T>::store(xn_p, e, cnt, VEC, yv);
                if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, VEC, pr);
            }
        }
    }
};

// Programmatic dependent launch: the dependent grid may start once every CTA
// of this grid has issued launch_dependents; griddepcontrol.wait blocks until
// the prerequisite grid has completed and its writes are visible.
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }


// Quotient by a divisor fixed for a launch, as a multiply-high and a shift
// (Granlund and Montgomery, division by invariant integers using
// multiplication): with l = ceil(log2 d) and m = floor(2^32 (2^l - d) / d) + 1,
// n / d = (umulhi(m, n) + n) >> l for 0 <= n < 2^31.  The CTAs of a launch
// split their block index into (asset, view, tile, channel group, ...) with
// these instead of integer divisions.
struct FastDiv {
    uint32_t d, m, l;
    __device__ __forceinline__ uint32_t quo(uint32_t n) const { return (__umulhi(m, n) + n) >> l; }
};
static FastDiv make_fastdiv(uint32_t d) {
    FastDiv f{d, 0u, 0u};
    while ((1ull << f.l) < d) ++f.l;
    f.m = (uint32_t)(((1ull << 32) * ((1ull << f.l) - d)) / d + 1);
    return f;
}

// Grid shape of a sparse step's launches and the divisors that split it.
struct SparseGrid {
    int n_cg, n_tiles, n_slices, n_stream, n_total;
    int small;  // n_total * n_stream < 2^31: the interleave's quotients in 32 bits
    FastDiv cg, tiles, a, na, slices, total;
};

// Tile offset i of the sparse form clamped to the records that exist, [0,
// cap]: a build whose records overflowed the capacity or the int32 offsets
// is flagged in the status word, and the transport then reads only records
// that exist.
__device__ __forceinline__ int record_offset(const int32_t* __restrict__ tile_ptr, size_t i, long long cap) {
    const long long x = __ldg(tile_ptr + i);
    return (int)(x < 0 ? 0 : (x < cap ? x : cap));
}

// Records of one pair applied by one CTA slice (grid-stride over the pair's
// records), channels [cg, cg + 4).  COPY: the value-copy ablation (no x0(t-1)
// gathers).
template <int K, bool COPY>
__device__ __forceinline__ void apply_records(const TransportArgs& args, const SparseGrid& g, int pair_id, int slice,
                                              int cg) {
    const int N = args.N, C = args.C, a = args.a;
    const int HW = args.H * args.W;
    const int T = g.n_tiles;
    const int n_slices = g.n_slices;
    const int pa = (int)g.a.quo((uint32_t)pair_id);
    const int s2 = pair_id - pa * a;
    const int b = (int)g.na.quo((uint32_t)pa);
    const int vi = pa - b * (N - a);
    const int v = args.others[vi];
    const int u = args.anchors[s2];
    const size_t pair = ((size_t)b * N + v) * N + u;
    const long long cap = args.max_records;
    const int r0 = record_offset(args.tile_ptr, pair * T, cap);
    const int r1 = record_offset(args.tile_ptr, pair * T + T, cap);
    const size_t plane = (size_t)HW;
    const float* xn = args.x0_new + ((size_t)b * a + s2) * C * plane;
    const float* xp = args.x0_prev + ((size_t)b * N + u) * C * plane;
    for (int r = r0 + slice * kThreads + threadIdx.x; r < r1; r += n_slices * kThreads) {
        const int4 rec = __ldg(reinterpret_cast<const int4*>(args.records) + r);
        Taps tp;
        taps_from_record<K>((int)((uint32_t)rec.x >> 28), rec.y, __int_as_float(rec.z), __int_as_float(rec.w),
                            args.W, tp);
        float* out = args.workspace + (size_t)r * C;
        {
            const int cn = C - cg < 4 ? C - cg : 4;
            float dn[K][4], dp[K][4];
#pragma unroll
            for (int kk = 0; kk < K; ++kk)
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    dn[kk][c] = 0.0f;
                    dp[kk][c] = 0.0f;
                    if (tp.q[kk] >= 0 && c < cn) {
                        const size_t e = (size_t)(cg + c) * plane + tp.q[kk];
                        dn[kk][c] = __ldg(xn + e);
                        if (!COPY) dp[kk][c] = __ldg(xp + e);
                    }
                }
            float g[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float acc = 0.0f;
#pragma unroll
                for (int kk = 0; kk < K; ++kk)
                    if (tp.q[kk] >= 0) acc = tap_term(COPY, tp.w[kk], dn[kk][c], dp[kk][c], acc);
                g[c] = acc;
            }
            if (cn == 4 && C % 4 == 0) {
                *reinterpret_cast<float4*>(out + cg) = make_float4(g[0], g[1], g[2], g[3]);
            } else {
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    if (c < cn) out[cg + c] = g[c];
            }
        }
    }
}

// Phase A: n_apply record-slice CTAs and n_stream anchor-view CTAs (tiles of
// kTileTokens tokens), each for one group of 4 channels, interleaved evenly in
// block order.
// Resident CTAs per SM the phases are compiled for, by latent type: with
// bf16 latents 6 (phase A, at most 40 registers) and 5 (phase B) put more
// gathers and streamed rows in flight than the few spilled registers cost
// (measured: unbounded, 62 / 56 registers, was 2-3 us slower per step); f32
// latents need more registers per quad and are left unbounded.
template <typename T>
constexpr int kPhaseABlocks = sizeof(T) == 2 ? 6 : 1;
template <typename T>
constexpr int kPhaseBBlocks = sizeof(T) == 2 ? 5 : 1;
// The increment-plane kernels (wide latents): phase A at 4 resident CTAs per
// SM (62 registers; at 5 or 6 its spills cost more than the residency
// gains), phase B at 5 (46 registers, no spills: it loads its streamed rows
// after the fold, so they are not held across the gathers; 4 or 6 resident
// CTAs, or the rows prefetched into the L2 before the wait, were slower).
constexpr int kPlaneABlocks = 4;
constexpr int kPlaneBBlocks = 5;

template <typename T, int K, bool VEC, bool COPY>
__global__ void __launch_bounds__(kThreads, kPhaseABlocks<T>) sparse_phase_a_kernel(const TransportArgs args,
                                                                                    const SparseGrid g) {
    pdl_launch_dependents();
    const uint32_t k = blockIdx.x;
    int s_before, s_next;
    if (g.small) {
        s_before = (int)g.total.quo(k * (uint32_t)g.n_stream);
        s_next = (int)g.total.quo((k + 1) * (uint32_t)g.n_stream);
    } else {
        s_before = (int)((long long)k * g.n_stream / g.n_total);
        s_next = (int)(((long long)k + 1) * g.n_stream / g.n_total);
    }
    if (s_next == s_before) {  // a record-apply CTA
        const int ai = (int)k - s_before;
        const int aj = (int)g.cg.quo((uint32_t)ai);
        const int pair = (int)g.slices.quo((uint32_t)aj);
        apply_records<K, COPY>(args, g, pair, aj - pair * g.n_slices, (ai - aj * g.n_cg) * 4);
        return;
    }
    const int q1 = (int)g.cg.quo((uint32_t)s_before);
    const int cg = (s_before - q1 * g.n_cg) * 4;
    const int q2 = (int)g.tiles.quo((uint32_t)q1);
    const int tile = q1 - q2 * g.n_tiles;
    const int b = (int)g.a.quo((uint32_t)q2);
    const int slot = q2 - b * args.a;
    const int v = args.anchors[slot];
    const int HW = args.H * args.W;
    const int tile0 = tile * kTileTokens;
    const int p0 = tile0 + 4 * threadIdx.x;
    if (p0 >= HW) return;
    const int cnt = HW - p0 < 4 ? HW - p0 : 4;
    const int cn = args.C - cg < 4 ? args.C - cg : 4;
    QuadRows<T, VEC> q;
    q.load(args, b, v, slot, p0, cnt, cg, cn);
    q.store(args, b, v, p0, cnt, cg, cn);
}

// Phase B: one CTA per (tile, group of 4 channels) of a view; blockIdx.y <
// N - a: views outside the anchor set (fold the tile's increments);
// blockIdx.y >= N - a: anchor views (only for an in-place cache update, see
// phase A).  PK = 0: each record's increment is its workspace row, written
// by phase A's apply; PK = K: it is formed here from the anchors' increment
// plane, sum_k w_k increment[q_k] in tap order (the same terms in the same
// order as the applies, so the same bits).
template <typename T, bool VEC, bool COPY, int PK>
__global__ void __launch_bounds__(kThreads, PK ? kPlaneBBlocks : kPhaseBBlocks<T>) sparse_phase_b_kernel(const TransportArgs args, const SparseGrid g) {
    __shared__ float s_acc[kTileTokens][4];
    __shared__ __align__(4) uint8_t s_n[kTileTokens];
    __shared__ int s_r0[GEOCACHE_MAX_VIEWS], s_cnt[GEOCACHE_MAX_VIEWS];
    const int HW = args.H * args.W;
    const int T_tiles = tiles_per_view_dev(args.H, args.W);
    const int n_cg = g.n_cg;
    const int tile = (int)g.cg.quo(blockIdx.x), cg = ((int)blockIdx.x - tile * n_cg) * 4, b = blockIdx.z;
    const int N = args.N, C = args.C, a = args.a;
    const int cn = C - cg < 4 ? C - cg : 4;
    const int tile0 = tile * kTileTokens;
    const int t = threadIdx.x;
    const int p0 = tile0 + 4 * t;
    const int cnt = p0 < HW ? (HW - p0 < 4 ? HW - p0 : 4) : 0;
    if ((int)blockIdx.y >= N - a) {  // anchor view, in-place update: after phase A's gathers
        const int slot = blockIdx.y - (N - a);
        pdl_wait();
        if (cnt <= 0) return;
        QuadRows<T, VEC> q;
        q.load(args, b, args.anchors[slot], slot, p0, cnt, cg, cn);
        q.store(args, b, args.anchors[slot], p0, cnt, cg, cn);
        return;
    }
    const int v = args.others[blockIdx.y];
    // streamed rows first (phase A writes none of them), tile offsets next;
    // with the plane (PK) the rows are loaded after the fold instead, which
    // keeps the fold's registers free for more resident CTAs
    QuadRows<T, VEC> q;
    if (!PK && cnt > 0) q.load(args, b, v, -1, p0, cnt, cg, cn);
    if (t < a) {
        const size_t i = (((size_t)b * N + v) * N + args.anchors[t]) * T_tiles + tile;
        // ranges clamped to the records that exist (an overflow is reported by the build)
        const int r0 = record_offset(args.tile_ptr, i, args.max_records);
        s_r0[t] = r0;
        s_cnt[t] = record_offset(args.tile_ptr, i + 1, args.max_records) - r0;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // the sums, cleared before the wait
        *reinterpret_cast<float4*>(s_acc[4 * t + i]) = make_float4(0.f, 0.f, 0.f, 0.f);
        s_n[4 * t + i] = 0;
    }
    __syncthreads();
    int total = 0;
    for (int s2 = 0; s2 < a; ++s2) total += s_cnt[s2];
    // a tile without records keeps x0(t-1) and reads and writes nothing phase A
    // touches (rows of views outside the anchor set), so it is stored without
    // waiting for phase A; the first CTA always waits, so that this grid
    // completes only after phase A
    const bool first = blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0;
    if (total == 0 && !first) {
        if (cnt > 0) {
            if (PK) q.load(args, b, v, -1, p0, cnt, cg, cn);
            q.store(args, b, v, p0, cnt, cg, cn);
        }
        return;
    }
    pdl_wait();  // phase A's workspace writes are complete and visible
    if (total == 0) {  // no record in the tile: every token keeps x0(t-1), nothing to fold
        if (cnt > 0) {
            if (PK) q.load(args, b, v, -1, p0, cnt, cg, cn);
            q.store(args, b, v, p0, cnt, cg, cn);
        }
        return;
    }
    for (int j0 = 0; j0 < total; j0 += kThreads) {
        const int j = j0 + t;
        int s_mine = -1, lp = 0;
        float g[4] = {0.f, 0.f, 0.f, 0.f};
        if (j < total) {
            int s2 = 0, jj = j;
            while (jj >= s_cnt[s2]) jj -= s_cnt[s2++];
            const int r = s_r0[s2] + jj;
            if (PK) {  // sum_k w_k increment[q_k] in tap order, from the anchor's increment plane
                const int4 rec = __ldg(reinterpret_cast<const int4*>(args.records) + r);
                lp = (rec.x & 0x0fffffff) - tile0;
                Taps tp;
                taps_from_record<PK ? PK : 1>((int)((uint32_t)rec.x >> 28), rec.y, __int_as_float(rec.z),
                                              __int_as_float(rec.w), args.W, tp);
                const float4* d = reinterpret_cast<const float4*>(args.workspace) +
                                  (((size_t)b * a + s2) * n_cg + cg / 4) * (size_t)HW;
                float4 dq[PK ? PK : 1];
#pragma unroll
                for (int kk = 0; kk < (PK ? PK : 1); ++kk)
                    dq[kk] = tp.q[kk] >= 0 ? __ldg(d + tp.q[kk]) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int kk = 0; kk < (PK ? PK : 1); ++kk) {
                    if (tp.q[kk] < 0) continue;
                    g[0] = __fmaf_rn(tp.w[kk], dq[kk].x, g[0]);
                    g[1] = __fmaf_rn(tp.w[kk], dq[kk].y, g[1]);
                    g[2] = __fmaf_rn(tp.w[kk], dq[kk].z, g[2]);
                    g[3] = __fmaf_rn(tp.w[kk], dq[kk].w, g[3]);
                }
            } else {
                lp = (__ldg(&args.records[r].token_mask) & 0x0fffffff) - tile0;
                const float* w = args.workspace + (size_t)r * C + cg;
                if (cn == 4 && C % 4 == 0) {
                    const float4 wq = *reinterpret_cast<const float4*>(w);
                    g[0] = wq.x; g[1] = wq.y; g[2] = wq.z; g[3] = wq.w;
                } else {
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        if (c < cn) g[c] = w[c];
                }
            }
            s_mine = s2;
        }
        // combine in anchor order (deterministic): anchor s2 adds in pass s2; the
        // records are in anchor order, so only the anchors of this round pass
        int s_lo = 0, c_lo = 0;
        while (c_lo + s_cnt[s_lo] <= j0) c_lo += s_cnt[s_lo++];
        const int j_last = (j0 + kThreads < total ? j0 + kThreads : total) - 1;
        int s_hi = s_lo, c_hi = c_lo;
        while (c_hi + s_cnt[s_hi] <= j_last) c_hi += s_cnt[s_hi++];
        for (int s2 = s_lo; s2 <= s_hi; ++s2) {
            if (s_mine == s2) {
                float4* dst = reinterpret_cast<float4*>(s_acc[lp]);
                float4 cur = *dst;
                cur.x = __fadd_rn(cur.x, g[0]);
                cur.y = __fadd_rn(cur.y, g[1]);
                cur.z = __fadd_rn(cur.z, g[2]);
                cur.w = __fadd_rn(cur.w, g[3]);
                *dst = cur;
                s_n[lp] += 1;
            }
            __syncthreads();
        }
    }
    if (cnt > 0) {
        if (PK) q.load(args, b, v, -1, p0, cnt, cg, cn);
        const uint32_t n4 = *reinterpret_cast<const uint32_t*>(s_n + 4 * t);
        if (n4) q.template fold4<COPY>(s_acc, n4, 4 * t);
        q.store(args, b, v, p0, cnt, cg, cn);
    }
}

// Phase A with the anchors' increment plane (wide latents): one CTA per
// (asset, anchor slot, tile, group of 4 channels) streams the anchor tile
// (x0(t) = x0_new and the reconstruction) and writes the tile's increment
// x0_new - x0(t-1) (x0_new itself under the value copy) to the plane
// [b][slot][channel group][token] x 4 channels in the workspace, where phase
// B gathers it at the records' taps.  Each element is read before the same
// thread writes it, so the stream is also correct for an in-place update.
template <typename T, bool VEC, bool COPY>
__global__ void __launch_bounds__(kThreads, kPlaneABlocks) sparse_phase_a_plane_kernel(const TransportArgs args,
                                                                                         const SparseGrid g) {
    pdl_launch_dependents();
    const int HW = args.H * args.W;
    const int n_cg = g.n_cg;
    const int q1 = (int)g.cg.quo(blockIdx.x);
    const int cgi = (int)blockIdx.x - q1 * n_cg;
    const int q2 = (int)g.tiles.quo((uint32_t)q1);
    const int tile = q1 - q2 * g.n_tiles;
    const int b = (int)g.a.quo((uint32_t)q2);
    const int slot = q2 - b * args.a;
    const int p0 = tile * kTileTokens + 4 * threadIdx.x;
    if (p0 >= HW) return;
    const int cnt = HW - p0 < 4 ? HW - p0 : 4;
    const int cg = cgi * 4;
    const int cn = args.C - cg < 4 ? args.C - cg : 4;
    const size_t plane = (size_t)HW;
    const int u = args.anchors[slot];
    const float* xn = args.x0_new + ((size_t)b * args.a + slot) * args.C * plane;
    const float* xp = args.x0_prev + ((size_t)b * args.N + u) * args.C * plane;
    const size_t view_base = ((size_t)b * args.N + u) * args.C * plane;
    const T* xt_p = static_cast<const T*>(args.x_t);
    T* xn_p = static_cast<T*>(args.x_next);
    float dn[4][4], pv[4][4];
    typename Lat4<T>::Raw xr[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        if (c >= cn) break;
        const size_t e = (size_t)(cg + c) * plane + p0;
        Lat4<float>::load(xn, e, cnt, VEC, dn[c]);
        if (!COPY) Lat4<float>::load(xp, e, cnt, VEC, pv[c]);
        if (args.coef.enabled) xr[c] = Lat4<T>::load_raw(xt_p, view_base + e, cnt, VEC);
    }
    float dd[4][4];
#pragma unroll
    for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int i = 0; i < 4; ++i) dd[c][i] = c < cn ? (COPY ? dn[c][i] : __fsub_rn(dn[c][i], pv[c][i])) : 0.0f;
    float4* d = reinterpret_cast<float4*>(args.workspace) + (((size_t)b * args.a + slot) * n_cg + cgi) * plane + p0;
#pragma unroll
    for (int i = 0; i < 4; ++i)
        if (i < cnt) d[i] = make_float4(dd[0][i], dd[1][i], dd[2][i], dd[3][i]);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        if (c >= cn) break;
        const size_t e = view_base + (size_t)(cg + c) * plane + p0;
        Lat4<float>::store(args.x0_out, e, cnt, VEC, dn[c]);
        if (args.coef.enabled) {
            float x[4], yv[4], pr[4];
            Lat4<T>::unpack(xr[c], x);
#pragma unroll
            for (int i = 0; i < 4; ++i) yv[i] = recon_one(args.coef, x[i], dn[c][i], pr[i]);
            Lat4<T>::store(xn_p, e, cnt, VEC, yv);
            if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, VEC, pr);
        }
    }
}

// Phase A by source tile (wide latents): one CTA per (asset, anchor slot,
// source tile, group of 4 channels).  It stages the anchor's increment
// x0_new - x0(t-1) (x0_new itself for the value copy) of the tile and of the
// W + 1 tokens after it in shared memory ([token][4 channels]: every tap of a
// record whose first kept tap lies in the tile), streams the anchor tile
// itself (x0(t) and the reconstruction) unless the update is in place, and
// then applies the tile's group of the source index: for each record whose
// target view is outside the anchor set, sum_k w_k increment[q_k] in tap
// order, read from shared memory, into its workspace row.  The scattered
// per-channel gathers of the record-parallel apply become one coalesced read
// of the anchor tile.
template <typename T, int K, bool COPY>
__global__ void __launch_bounds__(kThreads, kPhaseABlocks<T>) sparse_phase_a_src_kernel(const TransportArgs args,
                                                                                       const SparseGrid g, int stream) {
    pdl_launch_dependents();
    extern __shared__ __align__(16) float4 s_d[];  // [kTileTokens + W + 1] tokens x 4 channels
    const int HW = args.H * args.W, W = args.W;
    const int N = args.N, C = args.C, a = args.a;
    const int n_tiles = g.n_tiles;
    const int q1 = (int)g.cg.quo(blockIdx.x);
    const int cg = ((int)blockIdx.x - q1 * g.n_cg) * 4;
    const int q2 = (int)g.tiles.quo((uint32_t)q1);
    const int st = q1 - q2 * n_tiles;
    const int b = (int)g.a.quo((uint32_t)q2);
    const int slot = q2 - b * a;
    const int u = args.anchors[slot];
    const int cn = C - cg < 4 ? C - cg : 4;
    const size_t plane = (size_t)HW;
    const int tile0 = st * kTileTokens;
    const int span = min(kTileTokens + W + 1, HW - tile0);  // staged tokens
    const float* xn = args.x0_new + ((size_t)b * a + slot) * C * plane;
    const float* xp = args.x0_prev + ((size_t)b * N + u) * C * plane;
    const size_t view_base = ((size_t)b * N + u) * C * plane;
    const T* xt_p = static_cast<const T*>(args.x_t);
    T* xn_p = static_cast<T*>(args.x_next);
    const bool vec_rows = (HW & 3) == 0;
    for (int q = threadIdx.x; 4 * q < span; q += kThreads) {
        const int p0 = tile0 + 4 * q;
        const int cnt = min(4, span - 4 * q);
        const bool vec = vec_rows && cnt == 4;
        float dd[4][4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
#pragma unroll
            for (int i = 0; i < 4; ++i) dd[c][i] = 0.0f;
            if (c >= cn) continue;
            float dn[4];
            f4_load_keep(xn, (size_t)(cg + c) * plane + p0, cnt, vec, dn);
            if (!COPY) {
                float pv[4];
                f4_load_keep(xp, (size_t)(cg + c) * plane + p0, cnt, vec, pv);
#pragma unroll
                for (int i = 0; i < 4; ++i) dd[c][i] = __fsub_rn(dn[i], pv[i]);
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) dd[c][i] = dn[i];
            }
            if (stream && 4 * q < kTileTokens) {  // the anchor tile itself: x0(t) and the reconstruction
                const size_t e = view_base + (size_t)(cg + c) * plane + p0;
                Lat4<float>::store(args.x0_out, e, cnt, vec, dn);
                if (args.coef.enabled) {
                    float x[4], yv[4], pr[4];
                    Lat4<T>::load(xt_p, e, cnt, vec, x);
#pragma unroll
                    for (int i = 0; i < 4; ++i) yv[i] = recon_one(args.coef, x[i], dn[i], pr[i]);
                    Lat4<T>::store(xn_p, e, cnt, vec, yv);
                    if (args.pred_out) Lat4<float>::store(args.pred_out, e, cnt, vec, pr);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (i < cnt) s_d[4 * q + i] = make_float4(dd[0][i], dd[1][i], dd[2][i], dd[3][i]);
    }
    __syncthreads();
    const size_t grp = ((size_t)b * N + u) * n_tiles + st;  // group ends: see src_index_kernel
    const int lo = grp ? __ldg(args.src_ptr + grp - 1) : 0, hi = __ldg(args.src_ptr + grp);
    const int2* src_rec = reinterpret_cast<const int2*>(args.src_rec);
    for (int e0 = lo + threadIdx.x; e0 < hi; e0 += 2 * kThreads) {
        // two entries per thread, their loads in flight together
        int2 ent[2];
        int4 rec[2];
#pragma unroll
        for (int m = 0; m < 2; ++m) {
            const int e = e0 + m * kThreads;
            ent[m] = e < hi ? __ldg(src_rec + e) : make_int2(-1, 0);
            if (ent[m].x >= 0 && args.slot_of[ent[m].y] >= 0) ent[m].x = -1;  // target view is an anchor
            rec[m] = ent[m].x >= 0 ? __ldg(reinterpret_cast<const int4*>(args.records) + ent[m].x)
                                   : make_int4(0, 0, 0, 0);
        }
#pragma unroll
        for (int m = 0; m < 2; ++m) {
            if (ent[m].x < 0) continue;
            Taps tp;
            taps_from_record<K>((int)((uint32_t)rec[m].x >> 28), rec[m].y, __int_as_float(rec[m].z),
                                __int_as_float(rec[m].w), W, tp);
            float g[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int kk = 0; kk < K; ++kk) {
                if (tp.q[kk] < 0) continue;
                const float4 d = s_d[tp.q[kk] - tile0];
                g[0] = __fmaf_rn(tp.w[kk], d.x, g[0]);
                g[1] = __fmaf_rn(tp.w[kk], d.y, g[1]);
                g[2] = __fmaf_rn(tp.w[kk], d.z, g[2]);
                g[3] = __fmaf_rn(tp.w[kk], d.w, g[3]);
            }
            float* out = args.workspace + (size_t)ent[m].x * C + cg;
            if (cn == 4 && C % 4 == 0) {
                *reinterpret_cast<float4*>(out) = make_float4(g[0], g[1], g[2], g[3]);
            } else {
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    if (c < cn) out[c] = g[c];
            }
        }
    }
}

// The source-tile apply serves wide latents (at least kSrcMinChannels
// channels) whose workspace has no room for the increment plane, where the
// record-parallel apply's per-channel gathers dominate phase A; with few
// channels it is slower (it reads the anchors' whole x0(t-1) rows instead of
// the tapped tokens).
constexpr int kSrcMinChannels = 8;
// Record-parallel apply: CTAs per (pair, channel group) sized for about this
// many records each, from the mean records per ordered view pair.
constexpr long long kApplyRecords = 384;

template <typename T, int K>
static cudaError_t launch_sparse(const TransportArgs& t, cudaStream_t s) {
    const int HW = t.H * t.W;
    const int n_tiles = (HW + kTileTokens - 1) / kTileTokens;
    const int n_cg = (t.C + 3) / 4;
    const uintptr_t al = (uintptr_t)t.x0_new | (uintptr_t)t.x0_prev | (uintptr_t)t.x0_out | (uintptr_t)t.x_t |
                         (uintptr_t)t.x_next | (uintptr_t)t.pred_out;
    const bool vec = (HW % 4 == 0) && (al % 16 == 0);
    const bool in_place = t.x0_out == t.x0_prev;
    const bool copy = t.update == GEOCACHE_UPDATE_COPY;
    // wide latents: the anchors' increment plane when the workspace holds it
    // beside max_records * C floats, else phase A by source tile when the
    // corr has a source index and the staged span (tile + W + 1 tokens)
    // fits, else the record-parallel apply
    SparseGrid sg{};
    sg.n_cg = n_cg;
    sg.n_tiles = n_tiles;
    sg.cg = make_fastdiv((uint32_t)n_cg);
    sg.tiles = make_fastdiv((uint32_t)n_tiles);
    sg.a = make_fastdiv((uint32_t)t.a);
    sg.na = make_fastdiv((uint32_t)(t.N > t.a ? t.N - t.a : 1));
    const long long n_plane = plane_floats(t.B, t.a, t.C, HW);
    const bool by_plane = t.a < t.N && t.C >= kPlaneMinChannels && t.workspace &&
                          t.workspace_floats >= t.max_records * (long long)t.C + n_plane;
    const bool by_source = !by_plane && t.a < t.N && t.src_ptr && t.src_rec && t.C >= kSrcMinChannels &&
                           t.W + 1 <= kTileTokens;
    bool phase_a = false;
    if (by_plane) {
        const long long g = (long long)t.B * t.a * n_tiles * n_cg;
        if (g > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
        if (vec && !copy) sparse_phase_a_plane_kernel<T, true, false><<<(unsigned)g, kThreads, 0, s>>>(t, sg);
        else if (vec) sparse_phase_a_plane_kernel<T, true, true><<<(unsigned)g, kThreads, 0, s>>>(t, sg);
        else if (!copy) sparse_phase_a_plane_kernel<T, false, false><<<(unsigned)g, kThreads, 0, s>>>(t, sg);
        else sparse_phase_a_plane_kernel<T, false, true><<<(unsigned)g, kThreads, 0, s>>>(t, sg);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        phase_a = true;
    } else if (by_source) {
        const long long g = (long long)t.B * t.a * n_tiles * n_cg;
        if (g > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
        const size_t dyn = (size_t)(kTileTokens + t.W + 1) * sizeof(float4);
        if (!copy)
            sparse_phase_a_src_kernel<T, K, false><<<(unsigned)g, kThreads, dyn, s>>>(t, sg, in_place ? 0 : 1);
        else
            sparse_phase_a_src_kernel<T, K, true><<<(unsigned)g, kThreads, dyn, s>>>(t, sg, in_place ? 0 : 1);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        phase_a = true;
    } else {
        // apply CTAs per (pair, channel group): about kApplyRecords records each
        const long long pairs = (long long)t.B * t.N * (t.N - 1);
        const long long per_pair = (t.max_records + pairs - 1) / pairs;
        long long n_slices = (per_pair + kApplyRecords - 1) / kApplyRecords;
        n_slices = n_slices < 1 ? 1 : (n_slices > 64 ? 64 : n_slices);
        const long long n_apply = t.a < t.N ? (long long)t.B * (t.N - t.a) * t.a * n_slices * n_cg : 0;
        const long long n_stream = in_place ? 0 : (long long)t.B * t.a * n_tiles * n_cg;
        if (n_apply + n_stream > 0) {
            if (n_apply + n_stream > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
            const unsigned g = (unsigned)(n_apply + n_stream);
            sg.n_slices = (int)n_slices;
            sg.slices = make_fastdiv((uint32_t)n_slices);
            sg.n_stream = (int)n_stream;
            sg.n_total = (int)g;
            sg.total = make_fastdiv(g);
            sg.small = (long long)g * n_stream < 0x80000000LL;
            if (vec && !copy)
                sparse_phase_a_kernel<T, K, true, false><<<g, kThreads, 0, s>>>(t, sg);
            else if (vec)
                sparse_phase_a_kernel<T, K, true, true><<<g, kThreads, 0, s>>>(t, sg);
            else if (!copy)
                sparse_phase_a_kernel<T, K, false, false><<<g, kThreads, 0, s>>>(t, sg);
            else
                sparse_phase_a_kernel<T, K, false, true><<<g, kThreads, 0, s>>>(t, sg);
            cudaError_t e = cudaGetLastError();
            if (e != cudaSuccess) return e;
            phase_a = true;
        }
    }
    // an in-place update streams the anchor views after the wait, except with
    // the plane (its phase A reads each anchor element before writing it)
    const int gy = (t.N - t.a) + (in_place && !by_plane ? t.a : 0);
    if (gy > 0) {
        if ((long long)n_tiles * n_cg > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)(n_tiles * n_cg), gy, t.B);
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = 0;
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = phase_a ? 1 : 0;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        cudaError_t e;
        if (by_plane) {
            if (vec && !copy) e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, true, false, K>, t, sg);
            else if (vec) e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, true, true, K>, t, sg);
            else if (!copy) e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, false, false, K>, t, sg);
            else e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, false, true, K>, t, sg);
        } else {
            if (vec && !copy) e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, true, false, 0>, t, sg);
            else if (vec) e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, true, true, 0>, t, sg);
            else if (!copy) e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, false, false, 0>, t, sg);
            else e = cudaLaunchKernelEx(&cfg, sparse_phase_b_kernel<T, false, true, 0>, t, sg);
        }
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

// Persistent grid size of an instantiation: resident CTAs per SM x SMs.
template <typename Kern>
static int persistent_grid(Kern kern, size_t dyn_smem) {
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, dyn_smem) != cudaSuccess) return 0;
    return sms * (per_sm > 0 ? per_sm : 1);
}

template <typename T, int K, int MODE>
static cudaError_t launch_quad(const TransportArgs& t, cudaStream_t s) {
    const int HW = t.H * t.W;
    const uintptr_t al = (uintptr_t)t.x0_new | (uintptr_t)t.x0_prev | (uintptr_t)t.x0_out | (uintptr_t)t.x_t |
                         (uintptr_t)t.x_next | (uintptr_t)t.pred_out | (uintptr_t)t.keep | (uintptr_t)t.valid;
    const bool vec = (HW % 4 == 0) && (al % 16 == 0);
    const int n_tiles = (HW + kTileTokens - 1) / kTileTokens;
    const int n_cg = (t.C + 3) / 4;
    const long long n_units = (long long)t.B * t.N * n_tiles * n_cg;
    // TMA bulk rows need 16-byte aligned starts and sizes: HW % 8 == 0 covers bf16 rows
    if (vec && HW % 8 == 0) {
        TransportArgs ta = t;
        ta.wait_limit_ns = g_wait_limit_ns.load();
        ta.drop_first_copy = g_drop_first_copy.exchange(0);
        const size_t dyn = kStages * 4 * kTileTokens * (sizeof(float) + sizeof(T));
        auto kern = transport_fused_kernel<T, K, MODE>;
        static int grid = 0;  // per instantiation and process (one device per process)
        if (!grid) {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
            if (e != cudaSuccess) return e;
            grid = persistent_grid(kern, dyn);
            if (!grid) return cudaErrorInvalidConfiguration;
        }
        const long long g = n_units < grid ? n_units : grid;
        kern<<<(unsigned)g, kThreads, dyn, s>>>(ta, n_tiles, n_cg, n_units);
        return cudaGetLastError();
    }
    if (n_units > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    if (vec)
        transport_simple_kernel<T, K, MODE, true><<<(unsigned)n_units, kThreads, 0, s>>>(t, n_tiles, n_cg);
    else
        transport_simple_kernel<T, K, MODE, false><<<(unsigned)n_units, kThreads, 0, s>>>(t, n_tiles, n_cg);
    return cudaGetLastError();
}

template <typename T, int K>
static cudaError_t launch_transport_t(const TransportArgs& t, cudaStream_t s) {
    switch (t.mode) {
        case GEOCACHE_CORR_SPARSE: return launch_sparse<T, K>(t, s);
        case GEOCACHE_CORR_MASK: return launch_quad<T, K, GEOCACHE_CORR_MASK>(t, s);
        case GEOCACHE_CORR_TABLE: return launch_quad<T, K, GEOCACHE_CORR_TABLE>(t, s);
        default: return launch_quad<T, K, GEOCACHE_CORR_GEOMETRY>(t, s);
    }
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

// ------------------------------------------------- anchor-row pack / unpack --
// Gather (pack) of the anchor views' rows of a per-view tensor [B, N, row]
// into [B, a, row] in anchor order, and the scatter back (unpack): the batch
// slicing around the denoiser's anchor-only forward (Sec. 3.2).  Rows are
// copied as raw bytes, 16 bytes per thread when sizes and addresses allow.
template <int VB>
__global__ void __launch_bounds__(256) copy_rows_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                                        long long row_bytes, int N, int a, RowAnchors anc, int pack) {
    const int s = blockIdx.y, b = blockIdx.z;
    const int u = anc.v[s];
    const long long src_row = pack ? (long long)b * N + u : (long long)b * a + s;
    const long long dst_row = pack ? (long long)b * a + s : (long long)b * N + u;
    const uint8_t* sp = src + src_row * row_bytes;
    uint8_t* dp = dst + dst_row * row_bytes;
    const long long n = row_bytes / VB;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        if (VB == 16)
            __stcs(reinterpret_cast<uint4*>(dp) + i, __ldcs(reinterpret_cast<const uint4*>(sp) + i));
        else if (VB == 4)
            __stcs(reinterpret_cast<uint32_t*>(dp) + i, __ldcs(reinterpret_cast<const uint32_t*>(sp) + i));
        else
            dp[i] = sp[i];
    }
}

// ---------------------------------------------------- shuffled records --
// The shuffled-correspondence ablation (Sec. 4.3, "corr -> shuffled"): record
// r keeps its target token and takes the taps (keep mask, top-left tap,
// fractions) of record perm[r].  An entry outside [0, n) sets bit 2 of the
// status word and leaves the record as it was.
__global__ void __launch_bounds__(256) permute_records_kernel(const int4* __restrict__ src,
                                                              const int32_t* __restrict__ perm, int4* __restrict__ dst,
                                                              long long n) {
    for (long long r = blockIdx.x * (long long)blockDim.x + threadIdx.x; r < n; r += (long long)gridDim.x * blockDim.x) {
        const int4 own = __ldg(src + r);
        const int p = __ldg(perm + r);
        if (p < 0 || p >= n) {
            atomicOr(&g_device_error, 4u);
            dst[r] = own;
            continue;
        }
        const int4 o = __ldg(src + p);
        dst[r] = make_int4((int)(((uint32_t)own.x & 0x0fffffffu) | ((uint32_t)o.x & 0xf0000000u)), o.y, o.z, o.w);
    }
}

cudaError_t launch_permute_records(const geocache_tap_record* src, const int32_t* perm, geocache_tap_record* dst,
                                   long long n, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const long long blocks = (n + 255) / 256;
    permute_records_kernel<<<(unsigned)(blocks < 65535 * 8 ? blocks : 65535 * 8), 256, 0, s>>>(
        reinterpret_cast<const int4*>(src), perm, reinterpret_cast<int4*>(dst), n);
    return cudaGetLastError();
}

cudaError_t launch_copy_rows(const void* src, void* dst, long long row_bytes, int B, int N, int a,
                             const RowAnchors& anc, bool pack, cudaStream_t s) {
    if (row_bytes == 0 || B == 0 || a == 0) return cudaSuccess;
    const uintptr_t al = (uintptr_t)src | (uintptr_t)dst | (uintptr_t)row_bytes;
    const int vb = al % 16 == 0 ? 16 : (al % 4 == 0 ? 4 : 1);
    const long long n = row_bytes / vb;
    long long gx = (n + 255) / 256;
    if (gx > 1024) gx = 1024;
    dim3 grid((unsigned)gx, a, B);
    const uint8_t* sp = static_cast<const uint8_t*>(src);
    uint8_t* dp = static_cast<uint8_t*>(dst);
    if (vb == 16)
        copy_rows_kernel<16><<<grid, 256, 0, s>>>(sp, dp, row_bytes, N, a, anc, pack);
    else if (vb == 4)
        copy_rows_kernel<4><<<grid, 256, 0, s>>>(sp, dp, row_bytes, N, a, anc, pack);
    else
        copy_rows_kernel<1><<<grid, 256, 0, s>>>(sp, dp, row_bytes, N, a, anc, pack);
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

cudaError_t read_device_error(unsigned int* out, bool clear, cudaStream_t s) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(out, g_device_error, sizeof(unsigned int), 0, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return e;
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess || !clear || *out == 0) return e;
    static const unsigned int zero = 0;
    e = cudaMemcpyToSymbolAsync(g_device_error, &zero, sizeof(unsigned int), 0, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return e;
    return cudaStreamSynchronize(s);
}

}  // namespace geocache
