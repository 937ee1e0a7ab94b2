// Internal interface between the C ABI layer (geocache_api.cu) and the
// kernels (geocache_kernels.cu).  Not installed; not part of the ABI.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "geocache.h"

namespace geocache {

// Per-step sampler constants, formed in double on the host and rounded once.
struct ReconCoef {
    int enabled;     // 0: transport only
    int sampler;     // GEOCACHE_DDIM / GEOCACHE_FM_EULER
    int pred_kind;   // geocache_pred
    float st, s1t, inv_s1t, sp, s1p;   // DDIM: sqrt(ab_t), sqrt(1-ab_t), 1/sqrt(1-ab_t), sqrt(ab_prev), sqrt(1-ab_prev)
    float inv_sigma, dsigma;           // FM: 1/sigma, sigma_next - sigma
};

struct TransportArgs {
    int B, N, H, W, C, K, a;
    int c0, cn;                         // channel window [c0, c0 + cn) handled by this launch
    int mode;                           // geocache_corr_mode
    int write_anchor_rows;              // 0 when x0_out aliases x0_prev (rows written afterwards)
    int lat_dtype;                      // geocache_dtype
    int update;                         // geocache_update (Eq. 1 or the value-copy ablation)
    int drop_first_copy;                // test hook: unit 0's staged copies are not issued
    unsigned long long wait_limit_ns;   // limit of the bounded waits
    const float* pos;
    const uint8_t* valid;
    const geocache_camera* cams;
    const float* tau;
    const int32_t* idx;
    const float* w;
    const uint8_t* keep;
    const int32_t* tile_ptr;
    const geocache_tap_record* records;
    long long max_records;
    const int32_t* src_ptr;             // source index of the records (optional; see geocache_corr)
    const int32_t* src_rec;
    float* workspace;
    const float* x0_new;
    const float* x0_prev;
    float* x0_out;
    const void* x_t;
    void* x_next;
    float* pred_out;
    ReconCoef coef;
    int32_t anchors[GEOCACHE_MAX_VIEWS];
    int32_t slot_of[GEOCACHE_MAX_VIEWS];   // slot in `anchors`, -1 for non-anchors
    int32_t others[GEOCACHE_MAX_VIEWS];    // the views outside the anchor set, ascending
    long long workspace_floats;            // size of `workspace` (0 without one)
};

// The sparse step with wide latents (C >= kPlaneMinChannels) keeps the
// anchors' increments as a plane [b][anchor slot][channel group][token] x 4
// channels at the start of the workspace.  It takes that path only when the
// workspace holds max_records * C floats plus the plane, so that a minimal
// workspace keeps the per-record rows (see geocache_transport_workspace).
constexpr int kPlaneMinChannels = 8;
inline long long plane_floats(long long B, long long a, int C, long long HW) {
    return B * a * (long long)((C + 3) / 4) * 4 * HW;
}

struct RowAnchors {
    int32_t v[GEOCACHE_MAX_VIEWS];
};
cudaError_t launch_copy_rows(const void* src, void* dst, long long row_bytes, int B, int N, int a,
                             const RowAnchors& anc, bool pack, cudaStream_t s);

cudaError_t launch_tau(const float* pos, const uint8_t* valid, int B, int N, int H, int W,
                       float tol_frac, float* tau, cudaStream_t s);
cudaError_t launch_build_corr(const geocache_corr& c, cudaStream_t s);
// sparse form: per-tile record counts and their exclusive prefix sum in
// tile_ptr (tile_ptr[n] = total, or -1 when the total exceeds INT32_MAX)
cudaError_t launch_tile_ptr(const geocache_corr& c, cudaStream_t s);
cudaError_t launch_fill_records(const geocache_corr& c, cudaStream_t s);
// source index of the records (c.src_ptr, c.src_rec), after the records
cudaError_t launch_src_index(const geocache_corr& c, cudaStream_t s);
cudaError_t launch_permute_records(const geocache_tap_record* src, const int32_t* perm, geocache_tap_record* dst,
                                   long long n, cudaStream_t s);
__host__ __device__ int tiles_per_view(int H, int W);
cudaError_t launch_transport(const TransportArgs& t, cudaStream_t s);
cudaError_t launch_copy_anchor_rows(const TransportArgs& t, cudaStream_t s);
cudaError_t launch_reconstruct(const void* x_t, const float* x0, void* x_next, int lat_dtype, int64_t n,
                               const ReconCoef& coef, float* pred_out, float* x0_store, cudaStream_t s);

cudaError_t read_device_error(unsigned int* out, bool clear, cudaStream_t s);
// test hook of the bounded waits (geocache_debug_set_wait)
void set_debug_wait(unsigned long long limit_ns, int drop_first_copy);
cudaError_t read_raster_error(unsigned int* out, bool clear, cudaStream_t s);
// position maps at the token grid H x W; ss > 1: rendered at ss x H by
// ss x W (zbuf holds B*N*H*W*ss*ss words) and pooled to the token grid
cudaError_t launch_raster(const float* V, long long nv, const int32_t* F, long long nf, const int64_t* face_off,
                          int B, const geocache_camera* cams, int N, int H, int W, int ss, unsigned long long* zbuf,
                          float* pos, uint8_t* valid, cudaStream_t s);
cudaError_t launch_pool_posmaps(const float* pos_hi, const uint8_t* valid_hi, long long n_maps, int H, int W, int ss,
                                float* pos, uint8_t* valid, cudaStream_t s);

// Records a status and its message for geocache_last_error(); returns status.
int set_error(int status, const char* fmt, ...);

}  // namespace geocache
