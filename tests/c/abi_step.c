/*
 * A C caller of libgeocache.so (test support): one correspondence build and
 * one cached step with DDIM reconstruction through the plain C ABI, with
 * device memory from the CUDA runtime.
 *
 * usage: abi_step <input file> <output file>
 * input  (little-endian): int32 B, N, H, W, C; then float pos[B*N*H*W*3],
 *        uint8 valid[B*N*H*W], float cams[B*N*16], float x0_prev[B*N*C*H*W],
 *        float x_t[B*N*C*H*W], float delta[B*N*C*H*W] (the synthetic update
 *        of every view; the anchors' rows are used).
 * output: int32 anchors[2]; float tau[B], x0_out[B*N*C*H*W], x_next[B*N*C*H*W].
 * Exit status 0 when every call returned what the header promises.
 */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "geocache.h"

#define EXPECT(cond, ...)                              \
    do {                                               \
        if (!(cond)) {                                 \
            fprintf(stderr, "abi_step: " __VA_ARGS__); \
            fprintf(stderr, "\n");                     \
            return 1;                                  \
        }                                              \
    } while (0)

/* device buffer of `bytes`, filled from `host` (zeroed when host is NULL) */
static void* dev_copy(const void* host, size_t bytes) {
    void* d = NULL;
    if (cudaMalloc(&d, bytes ? bytes : 1) != cudaSuccess) return NULL;
    const cudaError_t e = host ? cudaMemcpy(d, host, bytes, cudaMemcpyHostToDevice) : cudaMemset(d, 0, bytes);
    return e == cudaSuccess ? d : NULL;
}

static int read_all(FILE* f, void* dst, size_t bytes) { return fread(dst, 1, bytes, f) == bytes; }

int main(int argc, char** argv) {
    EXPECT(argc == 3, "usage: abi_step <input> <output>");
    EXPECT(geocache_abi_version() == GEOCACHE_ABI_VERSION, "ABI version %d, header %d", geocache_abi_version(),
           GEOCACHE_ABI_VERSION);
    FILE* in = fopen(argv[1], "rb");
    EXPECT(in, "cannot open %s", argv[1]);
    int32_t dims[5];
    EXPECT(read_all(in, dims, sizeof dims), "short header");
    const int B = dims[0], N = dims[1], H = dims[2], W = dims[3], C = dims[4];
    const size_t tex = (size_t)B * N * H * W, lat = tex * C;
    float* pos = malloc(tex * 3 * 4);
    uint8_t* valid = malloc(tex);
    float* cams = malloc((size_t)B * N * 16 * 4);
    float* x0_prev = malloc(lat * 4);
    float* x_t = malloc(lat * 4);
    float* delta = malloc(lat * 4);
    EXPECT(pos && valid && cams && x0_prev && x_t && delta, "out of host memory");
    EXPECT(read_all(in, pos, tex * 12) && read_all(in, valid, tex) && read_all(in, cams, (size_t)B * N * 64) &&
               read_all(in, x0_prev, lat * 4) && read_all(in, x_t, lat * 4) && read_all(in, delta, lat * 4),
           "short input");
    fclose(in);

    /* anchors of the first cached step of a single-cached schedule */
    geocache_schedule sched;
    memset(&sched, 0, sizeof sched);
    sched.kind = GEOCACHE_SCHED_SINGLE_CACHED;
    int32_t anchors[2];
    int is_full = -1;
    EXPECT(geocache_rotate_anchors(N, 2, 1, 2, &sched, anchors, &is_full) == GEOCACHE_OK, "rotate: %s",
           geocache_last_error());
    EXPECT(is_full == 0, "step 1 of a single-cached schedule is cached");

    /* the anchors' denoiser x0: x0_prev + delta on their rows, [B, a, C, H, W] */
    const size_t row = (size_t)C * H * W;
    float* x0_new = malloc((size_t)B * 2 * row * 4);
    EXPECT(x0_new, "out of host memory");
    for (int b = 0; b < B; ++b)
        for (int s = 0; s < 2; ++s)
            for (size_t e = 0; e < row; ++e) {
                const size_t src = ((size_t)b * N + anchors[s]) * row + e;
                x0_new[((size_t)b * 2 + s) * row + e] = x0_prev[src] + delta[src];
            }

    float* d_pos = dev_copy(pos, tex * 12);
    uint8_t* d_valid = dev_copy(valid, tex);
    geocache_camera* d_cams = dev_copy(cams, (size_t)B * N * 64);
    float* d_tau = dev_copy(NULL, (size_t)B * 4);
    float* d_prev = dev_copy(x0_prev, lat * 4);
    float* d_new = dev_copy(x0_new, (size_t)B * 2 * row * 4);
    float* d_xt = dev_copy(x_t, lat * 4);
    float* d_out = dev_copy(NULL, lat * 4);
    float* d_xn = dev_copy(NULL, lat * 4);
    EXPECT(d_pos && d_valid && d_cams && d_tau && d_prev && d_new && d_xt && d_out && d_xn, "cudaMalloc failed");

    geocache_corr c;
    memset(&c, 0, sizeof c);
    c.B = B; c.N = N; c.H = H; c.W = W; c.K = 4;
    c.tol_frac = 0.01f;
    c.pos = d_pos; c.valid = d_valid; c.cams = d_cams; c.tau = d_tau;
    c.mode = GEOCACHE_CORR_GEOMETRY;
    EXPECT(geocache_build_corr(&c, NULL) == GEOCACHE_OK, "build: %s", geocache_last_error());

    geocache_recon r;
    memset(&r, 0, sizeof r);
    r.sampler = GEOCACHE_DDIM;
    r.a_t = 0.5;
    r.a_prev = 0.6;
    r.pred_kind = GEOCACHE_PRED_NONE;
    /* an argument error is reported before anything is launched */
    EXPECT(geocache_transport_step(&c, anchors, 0, C, d_new, d_prev, d_out, d_xt, d_xn, GEOCACHE_F32, &r, NULL, 0,
                                   NULL) == GEOCACHE_EINVAL, "a = 0 must be EINVAL");
    EXPECT(strlen(geocache_last_error()) > 0, "an error leaves a message");
    EXPECT(geocache_transport_step(&c, anchors, 2, C, d_new, d_prev, d_out, d_xt, d_xn, GEOCACHE_F32, &r, NULL, 0,
                                   NULL) == GEOCACHE_OK, "step: %s", geocache_last_error());
    EXPECT(cudaDeviceSynchronize() == cudaSuccess, "device error");
    EXPECT(geocache_device_status(NULL) == GEOCACHE_OK, "status: %s", geocache_last_error());

    float* tau = malloc((size_t)B * 4);
    float* x0_out = malloc(lat * 4);
    float* x_next = malloc(lat * 4);
    EXPECT(tau && x0_out && x_next, "out of host memory");
    EXPECT(cudaMemcpy(tau, d_tau, (size_t)B * 4, cudaMemcpyDeviceToHost) == cudaSuccess &&
               cudaMemcpy(x0_out, d_out, lat * 4, cudaMemcpyDeviceToHost) == cudaSuccess &&
               cudaMemcpy(x_next, d_xn, lat * 4, cudaMemcpyDeviceToHost) == cudaSuccess,
           "copy back failed");
    FILE* out = fopen(argv[2], "wb");
    EXPECT(out, "cannot open %s", argv[2]);
    EXPECT(fwrite(anchors, 4, 2, out) == 2 && fwrite(tau, 4, (size_t)B, out) == (size_t)B &&
               fwrite(x0_out, 4, lat, out) == lat && fwrite(x_next, 4, lat, out) == lat,
           "short write");
    fclose(out);
    printf("abi_step ok: anchors %d %d\n", anchors[0], anchors[1]);
    return 0;
}
