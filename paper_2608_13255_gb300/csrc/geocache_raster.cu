// Position-map rasteriser: the per-pixel world positions and validity masks
// that a geometry-conditioned texturing pipeline renders for each view
// (Sec. 3.1), from which the correspondence operator of Sec. 3.2 is built.
//
// A z-buffer over pixel centres, in two kernels:
//  raster_faces_kernel: one thread per face, looping over the views (the
//    face's vertices are loaded once; a CTA's faces normally belong to one
//    asset, whose cameras are staged in shared memory).  For each view the
//    face is projected; every pixel centre inside or on it (three
//    sign-normalised edge functions) gets the camera z of the ray /
//    face-plane intersection, and
//    the key (depth bits << 32 | face index) is min-combined into the
//    pixel's z-buffer word with a 64-bit atomicMin (nearest face wins, ties
//    to the lower face index; positive floats order like their bits).  The
//    pixel boxes of a warp's 32 faces are concatenated (prefix sums of the
//    box sizes) and the 32 lanes stride over the concatenation, each lane
//    finding its pixel's face by binary search over the prefix sums, so that
//    the work is balanced whatever the mix of small and large faces.
//  raster_resolve_kernel: one thread per pixel; the key's depth gives the
//    world position of the intersection.
// Super-sampled maps (the pipeline's image-resolution render brought to the
// latent token grid): the faces are rasterised at s times the token
// resolution with the cameras' focal lengths and principal point scaled by
// s, and raster_pool_kernel resolves each token's s x s pixels and pools
// them (mean of the valid pixels' positions, foreground when at least half
// are valid).  pool_posmaps_kernel pools maps the caller rendered itself.
// Every decision and the position are binary32 with one rounding per
// operation in a fixed order (explicit __f*_rn intrinsics), so the maps are
// reproducible bit for bit.
#include <cuda_runtime.h>

#include <cstdint>

#include "geocache.h"
#include "geocache_internal.h"

namespace geocache {

namespace {

// Status word of this translation unit (the library is linked without
// relocatable device code): bit 3 = a face index outside [0, nv).  Read and
// cleared together with the transport's word by geocache_device_status.
__device__ unsigned int g_raster_error = 0;

constexpr int kRasterThreads = 256;
constexpr unsigned long long kEmpty = ~0ull;  // z-buffer word of an uncovered pixel

struct Cam32 {
    float R[9], t[3], fx, fy, cx, cy;
};

// c points to global or shared memory (generic loads); the intrinsics are
// multiplied by `scale` (binary32), the camera of an s-times finer pixel grid
__device__ __forceinline__ Cam32 load_cam(const geocache_camera* c, float scale = 1.0f) {
    Cam32 k;
    const float* p = reinterpret_cast<const float*>(c);
#pragma unroll
    for (int i = 0; i < 9; ++i) k.R[i] = p[i];
#pragma unroll
    for (int i = 0; i < 3; ++i) k.t[i] = p[9 + i];
    k.fx = __fmul_rn(p[12], scale);
    k.fy = __fmul_rn(p[13], scale);
    k.cx = __fmul_rn(p[14], scale);
    k.cy = __fmul_rn(p[15], scale);
    return k;
}

// x_c = R X + t, each row summed ((R0 X0 + R1 X1) + R2 X2) + t
__device__ __forceinline__ void cam_point(const Cam32& c, const float (&X)[3], float* xc) {
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        float s = __fmul_rn(c.R[3 * r], X[0]);
        s = __fadd_rn(s, __fmul_rn(c.R[3 * r + 1], X[1]));
        s = __fadd_rn(s, __fmul_rn(c.R[3 * r + 2], X[2]));
        xc[r] = __fadd_rn(s, c.t[r]);
    }
}

// One projected face: screen vertices, signed area, camera-space plane
// n . x = nd, and the clamped pixel box.
struct Face {
    float u[3], v[3], area, n[3], nd;
    int ilo, ihi, jlo, jhi;
};

// A face of a warp published for the warp's balanced pixel loop.
struct FaceSlot {
    Face o;
    int b;           // asset
    unsigned int f;  // face index (low 32 bits of the z-buffer key)
};

// false when the face covers no pixel centre: a vertex not in front
// (z <= 1e-6), zero area, or a box outside the image
__device__ __forceinline__ bool setup_face(const Cam32& c, const float (&X)[3][3], int H, int W, Face& o) {
    float P[3][3];
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        cam_point(c, X[k], P[k]);
        if (!(P[k][2] > 1e-6f)) return false;
        o.u[k] = __fadd_rn(__fmul_rn(c.fx, __fdiv_rn(P[k][0], P[k][2])), c.cx);
        o.v[k] = __fadd_rn(__fmul_rn(c.fy, __fdiv_rn(P[k][1], P[k][2])), c.cy);
    }
    o.area = __fsub_rn(__fmul_rn(__fsub_rn(o.u[1], o.u[0]), __fsub_rn(o.v[2], o.v[0])),
                       __fmul_rn(__fsub_rn(o.v[1], o.v[0]), __fsub_rn(o.u[2], o.u[0])));
    if (!(o.area > 0.0f || o.area < 0.0f)) return false;
    const float umin = fminf(o.u[0], fminf(o.u[1], o.u[2])), umax = fmaxf(o.u[0], fmaxf(o.u[1], o.u[2]));
    const float vmin = fminf(o.v[0], fminf(o.v[1], o.v[2])), vmax = fmaxf(o.v[0], fmaxf(o.v[1], o.v[2]));
    const float ilo = fmaxf(ceilf(__fsub_rn(umin, 0.5f)), 0.0f), ihi = fminf(floorf(__fsub_rn(umax, 0.5f)), (float)(W - 1));
    const float jlo = fmaxf(ceilf(__fsub_rn(vmin, 0.5f)), 0.0f), jhi = fminf(floorf(__fsub_rn(vmax, 0.5f)), (float)(H - 1));
    if (!(ilo <= ihi && jlo <= jhi)) return false;
    o.ilo = (int)ilo;
    o.ihi = (int)ihi;
    o.jlo = (int)jlo;
    o.jhi = (int)jhi;
    float e1[3], e2[3];
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        e1[r] = __fsub_rn(P[1][r], P[0][r]);
        e2[r] = __fsub_rn(P[2][r], P[0][r]);
    }
    o.n[0] = __fsub_rn(__fmul_rn(e1[1], e2[2]), __fmul_rn(e1[2], e2[1]));
    o.n[1] = __fsub_rn(__fmul_rn(e1[2], e2[0]), __fmul_rn(e1[0], e2[2]));
    o.n[2] = __fsub_rn(__fmul_rn(e1[0], e2[1]), __fmul_rn(e1[1], e2[0]));
    float nd = __fmul_rn(o.n[0], P[0][0]);
    nd = __fadd_rn(nd, __fmul_rn(o.n[1], P[0][1]));
    o.nd = __fadd_rn(nd, __fmul_rn(o.n[2], P[0][2]));
    return true;
}

// camera-space ray direction through the pixel centre (pu, pv)
__device__ __forceinline__ void ray(const Cam32& c, float pu, float pv, float& d0, float& d1) {
    d0 = __fdiv_rn(__fsub_rn(pu, c.cx), c.fx);
    d1 = __fdiv_rn(__fsub_rn(pv, c.cy), c.fy);
}

// depth key of pixel (i, j) for the face, or kEmpty when its centre is not
// covered or the ray meets the plane at no positive finite depth
__device__ __forceinline__ unsigned long long pixel_key(const Cam32& c, const Face& o, int i, int j,
                                                        unsigned int face) {
    const float pu = __fadd_rn((float)i, 0.5f), pv = __fadd_rn((float)j, 0.5f);
    const float w0 = __fsub_rn(__fmul_rn(__fsub_rn(o.u[2], o.u[1]), __fsub_rn(pv, o.v[1])),
                               __fmul_rn(__fsub_rn(o.v[2], o.v[1]), __fsub_rn(pu, o.u[1])));
    const float w1 = __fsub_rn(__fmul_rn(__fsub_rn(o.u[0], o.u[2]), __fsub_rn(pv, o.v[2])),
                               __fmul_rn(__fsub_rn(o.v[0], o.v[2]), __fsub_rn(pu, o.u[2])));
    const float w2 = __fsub_rn(__fmul_rn(__fsub_rn(o.u[1], o.u[0]), __fsub_rn(pv, o.v[0])),
                               __fmul_rn(__fsub_rn(o.v[1], o.v[0]), __fsub_rn(pu, o.u[0])));
    const bool in = o.area > 0.0f ? (w0 >= 0.0f && w1 >= 0.0f && w2 >= 0.0f)
                                  : (w0 <= 0.0f && w1 <= 0.0f && w2 <= 0.0f);
    if (!in) return kEmpty;
    float d0, d1;
    ray(c, pu, pv, d0, d1);
    float den = __fmul_rn(o.n[0], d0);
    den = __fadd_rn(den, __fmul_rn(o.n[1], d1));
    den = __fadd_rn(den, o.n[2]);
    if (den == 0.0f) return kEmpty;
    const float s = __fdiv_rn(o.nd, den);
    if (!(s > 0.0f && s <= 3.0e38f)) return kEmpty;
    return ((unsigned long long)__float_as_uint(s) << 32) | face;
}

// asset of face f: face_off[b] <= f < face_off[b + 1] (clamped to [0, B))
__device__ __forceinline__ int asset_of(const int64_t* __restrict__ face_off, int B, long long f) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(face_off + mid) <= f) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

__global__ void __launch_bounds__(kRasterThreads, 4) raster_faces_kernel(
    const float* __restrict__ V, long long nv, const int32_t* __restrict__ F, long long nf,
    const int64_t* __restrict__ face_off, int B, const geocache_camera* __restrict__ cams, int N, int H, int W,
    float scale, unsigned long long* __restrict__ zbuf) {
    __shared__ geocache_camera s_cam[GEOCACHE_MAX_VIEWS];
    __shared__ int s_asset[2];
    __shared__ FaceSlot s_slot[kRasterThreads];
    __shared__ long long s_excl[kRasterThreads];
    const long long f0 = blockIdx.x * (long long)kRasterThreads;
    const long long f = f0 + threadIdx.x;
    const int lane = threadIdx.x & 31;
    // the CTA's faces belong to one asset unless it straddles a boundary
    if (threadIdx.x == 0) s_asset[0] = asset_of(face_off, B, f0);
    if (threadIdx.x == 1) s_asset[1] = asset_of(face_off, B, min(f0 + kRasterThreads, nf) - 1);
    __syncthreads();
    const bool one_asset = s_asset[0] == s_asset[1];
    for (int i = threadIdx.x; i < N * 16; i += kRasterThreads)
        reinterpret_cast<float*>(s_cam)[i] = __ldg(reinterpret_cast<const float*>(cams + (size_t)s_asset[0] * N) + i);
    __syncthreads();
    int b = s_asset[0];
    bool ok = f < nf;
    float X[3][3];
    if (ok) {
        if (!one_asset) b = asset_of(face_off, B, f);
#pragma unroll
        for (int k = 0; k < 3; ++k) {
            const int32_t vi = __ldg(F + 3 * f + k);
            if (vi < 0 || vi >= nv) {
                atomicOr(&g_raster_error, 8u);
                ok = false;
                break;
            }
            X[k][0] = __ldg(V + 3 * (size_t)vi);
            X[k][1] = __ldg(V + 3 * (size_t)vi + 1);
            X[k][2] = __ldg(V + 3 * (size_t)vi + 2);
        }
    }
    FaceSlot* slots = s_slot + (threadIdx.x & ~31);
    long long* excl_w = s_excl + (threadIdx.x & ~31);
    for (int view = 0; view < N; ++view) {
        const Cam32 c = load_cam(b == s_asset[0] ? s_cam + view : cams + (size_t)b * N + view, scale);
        Face o;
        const bool live = ok && setup_face(c, X, H, W, o);
        const long long box = live ? (long long)(o.ihi - o.ilo + 1) * (o.jhi - o.jlo + 1) : 0;
        if (live) {
            FaceSlot& my = s_slot[threadIdx.x];
            my.o = o;
            my.b = b;
            my.f = (unsigned int)f;
        }
        // prefix sums of the warp's box sizes: lane l's pixels are [excl, excl + box)
        long long incl = box;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const long long y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += y;
        }
        const long long total = __shfl_sync(0xffffffffu, incl, 31);
        s_excl[threadIdx.x] = incl - box;
        __syncwarp();
        for (long long k = lane; k < total; k += 32) {
            // the face of pixel k: the last lane whose range starts at or before k
            // (it has a non-empty box, and k lies inside it)
            int src = 0;
#pragma unroll
            for (int step = 16; step > 0; step >>= 1)
                if (excl_w[src + step] <= k) src += step;
            const FaceSlot& q = slots[src];
            const int local = (int)(k - excl_w[src]);
            const int bw = q.o.ihi - q.o.ilo + 1;
            const int i = q.o.ilo + local % bw, j = q.o.jlo + local / bw;
            const Cam32 qc = load_cam(q.b == s_asset[0] ? s_cam + view : cams + (size_t)q.b * N + view, scale);
            const unsigned long long key = pixel_key(qc, q.o, i, j, q.f);
            if (key != kEmpty) atomicMin(zbuf + ((size_t)q.b * N + view) * (size_t)H * W + (size_t)j * W + i, key);
        }
        __syncwarp();  // the slots are rewritten for the next view
    }
}

// World position of the surface point of pixel (i, j) whose z-buffer key is
// `key` (not kEmpty): the ray through the pixel centre at the key's depth,
// x_w = R^T (x_c - t).
__device__ __forceinline__ void key_position(const Cam32& c, unsigned long long key, int i, int j, float (&X)[3]) {
    const float s = __uint_as_float((unsigned int)(key >> 32));
    float d0, d1;
    ray(c, __fadd_rn((float)i, 0.5f), __fadd_rn((float)j, 0.5f), d0, d1);
    const float xc[3] = {__fsub_rn(__fmul_rn(s, d0), c.t[0]), __fsub_rn(__fmul_rn(s, d1), c.t[1]),
                         __fsub_rn(s, c.t[2])};
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        float x = __fmul_rn(c.R[r], xc[0]);
        x = __fadd_rn(x, __fmul_rn(c.R[3 + r], xc[1]));
        X[r] = __fadd_rn(x, __fmul_rn(c.R[6 + r], xc[2]));
    }
}

__global__ void __launch_bounds__(kRasterThreads) raster_resolve_kernel(const unsigned long long* __restrict__ zbuf,
                                                                         const geocache_camera* __restrict__ cams,
                                                                         int N, int H, int W, long long n_pix,
                                                                         float* __restrict__ pos,
                                                                         uint8_t* __restrict__ valid) {
    const long long HW = (long long)H * W;
    for (long long p = blockIdx.x * (long long)kRasterThreads + threadIdx.x; p < n_pix;
         p += (long long)gridDim.x * kRasterThreads) {
        const unsigned long long key = zbuf[p];
        float X[3] = {0.0f, 0.0f, 0.0f};
        if (key != kEmpty) {
            const int pix = (int)(p % HW);
            key_position(load_cam(cams + p / HW), key, pix % W, pix / W, X);  // [B, N] cameras, one per map
        }
        pos[3 * p] = X[0];
        pos[3 * p + 1] = X[1];
        pos[3 * p + 2] = X[2];
        valid[p] = key != kEmpty;
    }
}

// Token (i, j) of a token-grid map from its s x s pixels (i s + sx, j s + sy)
// of the fine map: positions of the valid pixels summed componentwise in
// binary32, pixel rows sy ascending and sx ascending within a row, divided
// once by their number n; foreground when 2 n >= s * s.
struct PoolAcc {
    float sum[3] = {0.0f, 0.0f, 0.0f};
    int n = 0;
    __device__ __forceinline__ void add(const float (&X)[3]) {
#pragma unroll
        for (int c = 0; c < 3; ++c) sum[c] = __fadd_rn(sum[c], X[c]);
        ++n;
    }
    __device__ __forceinline__ void store(int s, float* __restrict__ pos, uint8_t* __restrict__ valid, long long p) const {
        const bool fg = n > 0 && 2 * n >= s * s;
#pragma unroll
        for (int c = 0; c < 3; ++c) pos[3 * p + c] = fg ? __fdiv_rn(sum[c], (float)n) : 0.0f;
        valid[p] = fg;
    }
};

// resolve + pool of a z-buffer rendered at s x the token grid: one thread per
// token, grid-stride over the B * N * H * W tokens
__global__ void __launch_bounds__(kRasterThreads) raster_pool_kernel(const unsigned long long* __restrict__ zbuf,
                                                                      const geocache_camera* __restrict__ cams,
                                                                      int H, int W, int s, long long n_tok,
                                                                      float* __restrict__ pos,
                                                                      uint8_t* __restrict__ valid) {
    const long long HW = (long long)H * W;
    const int Ws = W * s;
    for (long long p = blockIdx.x * (long long)kRasterThreads + threadIdx.x; p < n_tok;
         p += (long long)gridDim.x * kRasterThreads) {
        const long long map = p / HW;
        const int tok = (int)(p % HW), i = tok % W, j = tok / W;
        const unsigned long long* zmap = zbuf + map * HW * s * s;
        const Cam32 c = load_cam(cams + map, (float)s);
        PoolAcc acc;
        for (int sy = 0; sy < s; ++sy)
            for (int sx = 0; sx < s; ++sx) {
                const int I = i * s + sx, J = j * s + sy;
                const unsigned long long key = __ldg(zmap + (size_t)J * Ws + I);
                if (key == kEmpty) continue;
                float X[3];
                key_position(c, key, I, J, X);
                acc.add(X);
            }
        acc.store(s, pos, valid, p);
    }
}

// pool of fine maps given by the caller: pos_hi [n_maps, H s, W s, 3],
// valid_hi [n_maps, H s, W s] -> pos [n_maps, H, W, 3], valid [n_maps, H, W]
__global__ void __launch_bounds__(kRasterThreads) pool_posmaps_kernel(const float* __restrict__ pos_hi,
                                                                       const uint8_t* __restrict__ valid_hi,
                                                                       int H, int W, int s, long long n_tok,
                                                                       float* __restrict__ pos,
                                                                       uint8_t* __restrict__ valid) {
    const long long HW = (long long)H * W;
    const long long Ws = (long long)W * s;
    for (long long p = blockIdx.x * (long long)kRasterThreads + threadIdx.x; p < n_tok;
         p += (long long)gridDim.x * kRasterThreads) {
        const long long map = p / HW;
        const int tok = (int)(p % HW), i = tok % W, j = tok / W;
        const long long base = map * HW * s * s;
        PoolAcc acc;
        for (int sy = 0; sy < s; ++sy)
            for (int sx = 0; sx < s; ++sx) {
                const long long q = base + ((long long)j * s + sy) * Ws + (long long)i * s + sx;
                if (!__ldg(valid_hi + q)) continue;
                const float X[3] = {__ldg(pos_hi + 3 * q), __ldg(pos_hi + 3 * q + 1), __ldg(pos_hi + 3 * q + 2)};
                acc.add(X);
            }
        acc.store(s, pos, valid, p);
    }
}

}  // namespace

cudaError_t read_raster_error(unsigned int* out, bool clear, cudaStream_t s) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(out, g_raster_error, sizeof(unsigned int), 0, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return e;
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess || !clear || *out == 0) return e;
    static const unsigned int zero = 0;
    e = cudaMemcpyToSymbolAsync(g_raster_error, &zero, sizeof(unsigned int), 0, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return e;
    return cudaStreamSynchronize(s);
}

// grid of a grid-stride kernel over n items: at most 16 CTAs per SM
static unsigned stride_grid(long long n) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long long want = (n + kRasterThreads - 1) / kRasterThreads, cap = (long long)(sms > 0 ? sms : 1) * 16;
    return (unsigned)(want < cap ? (want > 0 ? want : 1) : cap);
}

cudaError_t launch_raster(const float* V, long long nv, const int32_t* F, long long nf, const int64_t* face_off,
                          int B, const geocache_camera* cams, int N, int H, int W, int ss, unsigned long long* zbuf,
                          float* pos, uint8_t* valid, cudaStream_t s) {
    const long long n_tok = (long long)B * N * H * W, n_pix = n_tok * ss * ss;
    cudaError_t e = cudaMemsetAsync(zbuf, 0xff, sizeof(unsigned long long) * (size_t)n_pix, s);
    if (e != cudaSuccess) return e;
    if (nf > 0) {
        const long long gx = (nf + kRasterThreads - 1) / kRasterThreads;
        if (gx > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
        raster_faces_kernel<<<(unsigned)gx, kRasterThreads, 0, s>>>(V, nv, F, nf, face_off, B, cams, N, H * ss,
                                                                    W * ss, (float)ss, zbuf);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (ss == 1)
        raster_resolve_kernel<<<stride_grid(n_pix), kRasterThreads, 0, s>>>(zbuf, cams, N, H, W, n_pix, pos, valid);
    else
        raster_pool_kernel<<<stride_grid(n_tok), kRasterThreads, 0, s>>>(zbuf, cams, H, W, ss, n_tok, pos, valid);
    return cudaGetLastError();
}

cudaError_t launch_pool_posmaps(const float* pos_hi, const uint8_t* valid_hi, long long n_maps, int H, int W, int ss,
                                float* pos, uint8_t* valid, cudaStream_t s) {
    const long long n_tok = n_maps * H * W;
    if (n_tok == 0) return cudaSuccess;
    pool_posmaps_kernel<<<stride_grid(n_tok), kRasterThreads, 0, s>>>(pos_hi, valid_hi, H, W, ss, n_tok, pos, valid);
    return cudaGetLastError();
}

}  // namespace geocache
