/*
 * Seeded-input generator: z-buffer rasteriser for triangle meshes.
 *
 * Produces the per-pixel world-space position map and validity mask that a
 * geometry-conditioned texturing pipeline renders for each view (the paper's
 * position maps, Sec. 3.1 and the correspondence-operator paragraph of
 * Sec. 3.2).  This file is INPUT GENERATION only: it holds none of the
 * method's arithmetic (no correspondence, transport or reconstruction).
 *
 * Camera convention (world -> camera): x_c = R x_w + t, +z forward, pixel
 * x to the right, pixel y down; pixel (i, j) has its centre at
 * (i + 0.5, j + 0.5).  The camera record is 16 floats:
 *   R[9] (row-major), t[3], fx, fy, cx, cy.
 *
 * The stored position of a covered pixel is the intersection of the ray
 * through the pixel centre with the plane of the nearest triangle whose
 * screen-space footprint contains that centre, computed in double precision
 * and rounded once to float.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

static void cam_load(const float* cam, double R[9], double t[3], double k[4]) {
    for (int i = 0; i < 9; ++i) R[i] = (double)cam[i];
    for (int i = 0; i < 3; ++i) t[i] = (double)cam[9 + i];
    for (int i = 0; i < 4; ++i) k[i] = (double)cam[12 + i];
}

/* Returns 0 on success, -1 on bad arguments, -2 on allocation failure. */
int synth_raster_mesh(const double* V, int nv, const int32_t* F, int nf,
                      const float* cam, int H, int W,
                      float* pos_out, uint8_t* valid_out) {
    if (!V || !F || !cam || !pos_out || !valid_out || nv <= 0 || nf < 0 || H <= 0 || W <= 0)
        return -1;
    double R[9], t[3], k[4];
    cam_load(cam, R, t, k);
    const double fx = k[0], fy = k[1], cx = k[2], cy = k[3];
    double* Vc = (double*)malloc(sizeof(double) * 3 * (size_t)nv);
    double* depth = (double*)malloc(sizeof(double) * (size_t)H * W);
    if (!Vc || !depth) { free(Vc); free(depth); return -2; }
    for (int i = 0; i < nv; ++i) {
        const double* p = V + 3 * (size_t)i;
        for (int r = 0; r < 3; ++r)
            Vc[3 * (size_t)i + r] = R[3 * r] * p[0] + R[3 * r + 1] * p[1] + R[3 * r + 2] * p[2] + t[r];
    }
    for (size_t i = 0; i < (size_t)H * W; ++i) {
        depth[i] = INFINITY;
        valid_out[i] = 0;
        pos_out[3 * i] = pos_out[3 * i + 1] = pos_out[3 * i + 2] = 0.0f;
    }
    for (int f = 0; f < nf; ++f) {
        const int32_t a = F[3 * (size_t)f], b = F[3 * (size_t)f + 1], c = F[3 * (size_t)f + 2];
        if (a < 0 || b < 0 || c < 0 || a >= nv || b >= nv || c >= nv) continue;
        const double* P0 = Vc + 3 * (size_t)a;
        const double* P1 = Vc + 3 * (size_t)b;
        const double* P2 = Vc + 3 * (size_t)c;
        if (P0[2] <= 1e-6 || P1[2] <= 1e-6 || P2[2] <= 1e-6) continue;
        const double u0 = fx * P0[0] / P0[2] + cx, v0 = fy * P0[1] / P0[2] + cy;
        const double u1 = fx * P1[0] / P1[2] + cx, v1 = fy * P1[1] / P1[2] + cy;
        const double u2 = fx * P2[0] / P2[2] + cx, v2 = fy * P2[1] / P2[2] + cy;
        const double area = (u1 - u0) * (v2 - v0) - (v1 - v0) * (u2 - u0);
        if (area == 0.0) continue;
        double umin = fmin(u0, fmin(u1, u2)), umax = fmax(u0, fmax(u1, u2));
        double vmin = fmin(v0, fmin(v1, v2)), vmax = fmax(v0, fmax(v1, v2));
        int i_lo = (int)ceil(umin - 0.5), i_hi = (int)floor(umax - 0.5);
        int j_lo = (int)ceil(vmin - 0.5), j_hi = (int)floor(vmax - 0.5);
        if (i_lo < 0) i_lo = 0;
        if (j_lo < 0) j_lo = 0;
        if (i_hi > W - 1) i_hi = W - 1;
        if (j_hi > H - 1) j_hi = H - 1;
        if (i_lo > i_hi || j_lo > j_hi) continue;
        /* plane of the triangle in camera coordinates: n . X = n . P0 */
        const double e1[3] = {P1[0] - P0[0], P1[1] - P0[1], P1[2] - P0[2]};
        const double e2[3] = {P2[0] - P0[0], P2[1] - P0[1], P2[2] - P0[2]};
        const double n[3] = {e1[1] * e2[2] - e1[2] * e2[1], e1[2] * e2[0] - e1[0] * e2[2],
                             e1[0] * e2[1] - e1[1] * e2[0]};
        const double nd = n[0] * P0[0] + n[1] * P0[1] + n[2] * P0[2];
        for (int j = j_lo; j <= j_hi; ++j) {
            const double pv = j + 0.5;
            for (int i = i_lo; i <= i_hi; ++i) {
                const double pu = i + 0.5;
                /* edge functions, sign-normalised by the triangle's orientation */
                double w0 = ((u2 - u1) * (pv - v1) - (v2 - v1) * (pu - u1)) / area;
                double w1 = ((u0 - u2) * (pv - v2) - (v0 - v2) * (pu - u2)) / area;
                double w2 = 1.0 - w0 - w1;
                if (w0 < 0.0 || w1 < 0.0 || w2 < 0.0) continue;
                const double d[3] = {(pu - cx) / fx, (pv - cy) / fy, 1.0};
                const double den = n[0] * d[0] + n[1] * d[1] + n[2] * d[2];
                if (den == 0.0) continue;
                const double s = nd / den; /* camera-space depth along +z */
                if (!(s > 0.0)) continue;
                const size_t pix = (size_t)j * W + i;
                if (s >= depth[pix]) continue;
                depth[pix] = s;
                const double xc[3] = {s * d[0] - t[0], s * d[1] - t[1], s * d[2] - t[2]};
                /* world = R^T (x_c - t) */
                for (int r = 0; r < 3; ++r)
                    pos_out[3 * pix + r] = (float)(R[r] * xc[0] + R[3 + r] * xc[1] + R[6 + r] * xc[2]);
                valid_out[pix] = 1;
            }
        }
    }
    free(Vc);
    free(depth);
    return 0;
}
