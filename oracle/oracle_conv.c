/*
 * Plain fp64 CPU reference ("the oracle") for fused-tile execution of a CNN
 * front-end (MAFAT, Sec. 4).  TEST INFRASTRUCTURE ONLY: the product path
 * never links, loads or calls this file; only the tests, the smoke check and
 * the benchmark's CPU-baseline leg do.  It shares no code with the CUDA path.
 *
 * What it computes is the plain definition of the layers the paper fuses
 * (Sec. 2, Sec. 4): a convolution layer followed by folded batch-norm and
 * leaky ReLU, and a max-pool layer.  Feature maps are HWC (channels
 * innermost), weights are [Cout][Cin][k][k] (cross-correlation, as in every
 * CNN framework), everything in double precision (single precision in the
 * fp32 build, see ORACLE_REAL below):
 *
 *   acc[y][x][o] = sum_{c, ky, kx} w[o][c][ky][kx] * in[y*s+ky-p][x*s+kx-p][c]
 *                  (input outside the map counts as 0)
 *   z            = scale[o] * acc + bias[o]
 *   out          = z > 0 ? z : slope * z
 *
 *   pool[y][x][c] = max_{dy, dx < k} in[y*s+dy][x*s+dx][c]
 *
 * The sum runs over (c, ky, kx) in ascending order, in every function here,
 * so the tiled variant reproduces the full-map variant bit for bit.
 *
 * Fused tile partitioning (Sec. 3, Sec. 4) evaluates each layer only on a
 * rectangle ("region") of its output, reading a rectangle of its input.  The
 * *_region functions take the input region buffer with its origin in map
 * coordinates and compute an output rectangle; a read that falls inside the
 * map but outside the supplied region is a region-computation error and makes
 * the call return -1 without writing anything further.
 *
 * Loops over output rows are split over OpenMP threads when available; this
 * changes no summation order.
 */
#include <stddef.h>

/* Arithmetic type: double (the parity oracle), or float when built with
 * -DORACLE_REAL=float (the plain fp32 forward the method statement names, built
 * as a second library and used only to time the CPU baseline; the same loops). */
#ifndef ORACLE_REAL
#define ORACLE_REAL double
#endif
typedef ORACLE_REAL real_t;

#define IDX3(y, x, c, W, C) ((((size_t)(y)) * (size_t)(W) + (size_t)(x)) * (size_t)(C) + (size_t)(c))

/* Full-map convolution + folded BN + leaky ReLU.  Returns 0, or -1 on bad sizes. */
int oracle_conv_full(const real_t* in, int H, int W, int Cin,
                     const real_t* w, int Cout, int k, int stride, int pad,
                     const real_t* scale, const real_t* bias, real_t slope,
                     real_t* out)
{
    if (H <= 0 || W <= 0 || Cin <= 0 || Cout <= 0 || k <= 0 || stride <= 0 || pad < 0) return -1;
    int Ho = (H + 2 * pad - k) / stride + 1;
    int Wo = (W + 2 * pad - k) / stride + 1;
    if (Ho <= 0 || Wo <= 0) return -1;
#pragma omp parallel for schedule(dynamic, 1)
    for (int y = 0; y < Ho; ++y) {
        for (int x = 0; x < Wo; ++x) {
            for (int o = 0; o < Cout; ++o) {
                real_t acc = 0.0;
                for (int c = 0; c < Cin; ++c) {
                    for (int ky = 0; ky < k; ++ky) {
                        int iy = y * stride + ky - pad;
                        if (iy < 0 || iy >= H) continue;
                        for (int kx = 0; kx < k; ++kx) {
                            int ix = x * stride + kx - pad;
                            if (ix < 0 || ix >= W) continue;
                            real_t wv = w[(((size_t)o * Cin + c) * k + ky) * k + kx];
                            acc += wv * in[IDX3(iy, ix, c, W, Cin)];
                        }
                    }
                }
                real_t z = scale[o] * acc + bias[o];
                out[IDX3(y, x, o, Wo, Cout)] = z > 0.0 ? z : slope * z;
            }
        }
    }
    return 0;
}

/* Full-map max-pool (no padding).  Returns 0, or -1 on bad sizes. */
int oracle_maxpool_full(const real_t* in, int H, int W, int C, int k, int stride, real_t* out)
{
    if (H <= 0 || W <= 0 || C <= 0 || k <= 0 || stride <= 0 || H < k || W < k) return -1;
    int Ho = (H - k) / stride + 1;
    int Wo = (W - k) / stride + 1;
#pragma omp parallel for schedule(static)
    for (int y = 0; y < Ho; ++y)
        for (int x = 0; x < Wo; ++x)
            for (int c = 0; c < C; ++c) {
                real_t m = in[IDX3(y * stride, x * stride, c, W, C)];
                for (int dy = 0; dy < k; ++dy)
                    for (int dx = 0; dx < k; ++dx) {
                        real_t v = in[IDX3(y * stride + dy, x * stride + dx, c, W, C)];
                        if (v > m) m = v;
                    }
                out[IDX3(y, x, c, Wo, C)] = m;
            }
    return 0;
}

/*
 * Convolution evaluated on the output rectangle [oy0, oy0+oh) x [ox0, ox0+ow)
 * (map coordinates) from an input region buffer in[ih][iw][Cin] whose element
 * (0, 0) sits at map position (iy0, ix0) of a map of size mh x mw.
 * Output buffer is out[oh][ow][Cout].  Returns 0, or -1 if a needed in-map
 * input pixel is missing from the region (or on bad sizes).
 */
int oracle_conv_region(const real_t* in, int iy0, int ix0, int ih, int iw,
                       int mh, int mw, int Cin,
                       const real_t* w, int Cout, int k, int stride, int pad,
                       const real_t* scale, const real_t* bias, real_t slope,
                       int oy0, int ox0, int oh, int ow, real_t* out)
{
    if (ih < 0 || iw < 0 || oh < 0 || ow < 0 || Cin <= 0 || Cout <= 0 || k <= 0 || stride <= 0) return -1;
    /* Check first that every needed in-map pixel is in the region. */
    for (int y = oy0; y < oy0 + oh; ++y)
        for (int ky = 0; ky < k; ++ky) {
            int my = y * stride + ky - pad;
            if (my < 0 || my >= mh) continue;
            if (my < iy0 || my >= iy0 + ih) return -1;
        }
    for (int x = ox0; x < ox0 + ow; ++x)
        for (int kx = 0; kx < k; ++kx) {
            int mx = x * stride + kx - pad;
            if (mx < 0 || mx >= mw) continue;
            if (mx < ix0 || mx >= ix0 + iw) return -1;
        }
#pragma omp parallel for schedule(dynamic, 1)
    for (int yy = 0; yy < oh; ++yy) {
        int y = oy0 + yy;
        for (int xx = 0; xx < ow; ++xx) {
            int x = ox0 + xx;
            for (int o = 0; o < Cout; ++o) {
                real_t acc = 0.0;
                for (int c = 0; c < Cin; ++c) {
                    for (int ky = 0; ky < k; ++ky) {
                        int my = y * stride + ky - pad;
                        if (my < 0 || my >= mh) continue;
                        for (int kx = 0; kx < k; ++kx) {
                            int mx = x * stride + kx - pad;
                            if (mx < 0 || mx >= mw) continue;
                            real_t wv = w[(((size_t)o * Cin + c) * k + ky) * k + kx];
                            acc += wv * in[IDX3(my - iy0, mx - ix0, c, iw, Cin)];
                        }
                    }
                }
                real_t z = scale[o] * acc + bias[o];
                out[IDX3(yy, xx, o, ow, Cout)] = z > 0.0 ? z : slope * z;
            }
        }
    }
    return 0;
}

/* Max-pool evaluated on an output rectangle from an input region buffer (as above). */
int oracle_maxpool_region(const real_t* in, int iy0, int ix0, int ih, int iw,
                          int mh, int mw, int C, int k, int stride,
                          int oy0, int ox0, int oh, int ow, real_t* out)
{
    if (ih < 0 || iw < 0 || oh < 0 || ow < 0 || C <= 0 || k <= 0 || stride <= 0) return -1;
    for (int y = oy0; y < oy0 + oh; ++y)
        for (int dy = 0; dy < k; ++dy) {
            int my = y * stride + dy;
            if (my >= mh || my < iy0 || my >= iy0 + ih) return -1;
        }
    for (int x = ox0; x < ox0 + ow; ++x)
        for (int dx = 0; dx < k; ++dx) {
            int mx = x * stride + dx;
            if (mx >= mw || mx < ix0 || mx >= ix0 + iw) return -1;
        }
    for (int yy = 0; yy < oh; ++yy)
        for (int xx = 0; xx < ow; ++xx)
            for (int c = 0; c < C; ++c) {
                int by = (oy0 + yy) * stride - iy0, bx = (ox0 + xx) * stride - ix0;
                real_t m = in[IDX3(by, bx, c, iw, C)];
                for (int dy = 0; dy < k; ++dy)
                    for (int dx = 0; dx < k; ++dx) {
                        real_t v = in[IDX3(by + dy, bx + dx, c, iw, C)];
                        if (v > m) m = v;
                    }
                out[IDX3(yy, xx, c, ow, C)] = m;
            }
    return 0;
}

/* Number of OpenMP threads the loops above use (1 without OpenMP). */
int oracle_num_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Set the number of OpenMP threads of the loops above (n >= 1; no effect without OpenMP). */
void oracle_set_num_threads(int n)
{
#ifdef _OPENMP
    extern void omp_set_num_threads(int);
    if (n >= 1) omp_set_num_threads(n);
#else
    (void)n;
#endif
}
