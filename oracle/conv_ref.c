/*
 * Oracle direct convolution (TEST INFRASTRUCTURE ONLY).
 *
 * This file belongs to the CPU oracle of the carry-through checksum method
 * (Sec. II-A of the paper).  Only the tests, the smoke check and the CPU
 * baseline of the benchmark may load it; the product path never does.
 *
 * It computes the plain definition of a 2-D convolution of one image:
 *
 *     y[k][p][q] = sum over (c, r, s) with skip[k][c][r][s] == 0 of
 *                  w[k][c][r][s] * x[c][p*stride + r - pad][q*stride + s - pad]
 *
 * with zero padding, accumulating in IEEE double.  Weights whose skip flag is
 * set are structural zeros of the carry-through construction (the zero slice
 * that multiplies the incoming checksum channel, Sec. II-A "input-channel
 * level", and the off-centre taps of a carry-through filter, Fig. 1): they are
 * left out of the sum instead of being multiplied, so an infinite or NaN
 * checksum cannot leak into a data channel through 0 * inf.
 *
 * A fully-connected layer is the same routine with H = W = R = S = 1.
 *
 * The loops are the definition written out; the order of the (c, r, s) sum is
 * fixed (c outer, r, s inner) and the accumulation is in double, so results
 * do not depend on the thread count.  Build with -ffp-contract=off so that no
 * multiply-add is fused.
 */
#include <stddef.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

void or_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int or_get_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void or_conv2d(const double *x, int C, int H, int W,
               const double *w, const unsigned char *skip,
               int K, int R, int S, int stride, int pad,
               int P, int Q, double *y)
{
    long k;
#pragma omp parallel for schedule(dynamic, 1)
    for (k = 0; k < K; ++k) {
        double *yk = y + (size_t)k * P * Q;
        memset(yk, 0, sizeof(double) * (size_t)P * Q);
        for (int c = 0; c < C; ++c) {
            for (int r = 0; r < R; ++r) {
                for (int s = 0; s < S; ++s) {
                    size_t wi = (((size_t)k * C + c) * R + r) * S + s;
                    if (skip && skip[wi]) continue;
                    double wv = w[wi];
                    /* output columns q whose input column q*stride+s-pad lies in [0, W) */
                    int qlo = (pad - s > 0) ? (pad - s + stride - 1) / stride : 0;
                    int qhi = (W - 1 - s + pad >= 0) ? (W - 1 - s + pad) / stride + 1 : 0;
                    if (qhi > Q) qhi = Q;
                    for (int p = 0; p < P; ++p) {
                        int h = p * stride + r - pad;
                        if (h < 0 || h >= H) continue;
                        const double *xr = x + ((size_t)c * H + h) * W;
                        double *yr = yk + (size_t)p * Q;
                        if (stride == 1) {
                            for (int q = qlo; q < qhi; ++q) yr[q] += wv * xr[q + s - pad];
                        } else {
                            for (int q = qlo; q < qhi; ++q) yr[q] += wv * xr[q * stride + s - pad];
                        }
                    }
                }
            }
        }
    }
}
