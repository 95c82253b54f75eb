/*
 * CPU oracle: direct convolution on INT8 codes. TEST INFRASTRUCTURE ONLY.
 *
 * Only tests, the smoke check and the benchmark's CPU-baseline leg may load
 * this library. It shares no code with the CUDA path.
 *
 * Computes the integer accumulator of Eq. (integer_accumulation) with zero
 * points 0 (symmetric codes), for the convolution written as the unfolded
 * linear operator of Eq. (linear_operator): for each output pixel p and output
 * channel o,
 *     acc[p, o] = sum_{kh, kw, ci} x[p*stride + k - pad, ci] * w[o, kh, kw, ci]
 * with zero padding outside the input. Plain nested loops, int64 sums.
 *
 * x  : NHWC int8, shape [n][h][w][c]
 * wt : OHWI int8, shape [co][kh][kw][c]
 * acc: int64, shape [n][ho1-ho0][wo1-wo0][co] (an output window; the full
 *      output is ho0 = wo0 = 0, ho1 = Ho, wo1 = Wo)
 *
 * When built with OpenMP the output rows are shared among threads; every sum
 * is an exact integer, so the result does not depend on the thread count.
 */
#include <stdint.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Threads the direct convolution may use (1 without OpenMP). */
int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int t)
{
#ifdef _OPENMP
    if (t > 0) omp_set_num_threads(t);
#else
    (void)t;
#endif
}

void oracle_conv2d_codes(const int8_t *x, int64_t n, int64_t h, int64_t w, int64_t c,
                         const int8_t *wt, int64_t co, int64_t kh, int64_t kw,
                         int64_t stride, int64_t pad,
                         int64_t ho0, int64_t ho1, int64_t wo0, int64_t wo1,
                         int64_t *acc)
{
    int64_t nho = ho1 - ho0, nwo = wo1 - wo0;
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int64_t b = 0; b < n; ++b)
        for (int64_t oy = ho0; oy < ho1; ++oy)
            for (int64_t ox = wo0; ox < wo1; ++ox) {
                int64_t *out = acc + (((b * nho) + (oy - ho0)) * nwo + (ox - wo0)) * co;
                for (int64_t o = 0; o < co; ++o) {
                    int64_t s = 0;
                    for (int64_t ky = 0; ky < kh; ++ky) {
                        int64_t iy = oy * stride + ky - pad;
                        if (iy < 0 || iy >= h) continue;
                        for (int64_t kx = 0; kx < kw; ++kx) {
                            int64_t ix = ox * stride + kx - pad;
                            if (ix < 0 || ix >= w) continue;
                            const int8_t *xp = x + ((b * h + iy) * w + ix) * c;
                            const int8_t *wp = wt + ((o * kh + ky) * kw + kx) * c;
                            for (int64_t ci = 0; ci < c; ++ci)
                                s += (int64_t)xp[ci] * (int64_t)wp[ci];
                        }
                    }
                    out[o] = s;
                }
            }
}

/* The same sum at an explicit list of output pixels pix[i] = (b, oy, ox). */
void oracle_conv2d_codes_at(const int8_t *x, int64_t n, int64_t h, int64_t w, int64_t c,
                            const int8_t *wt, int64_t co, int64_t kh, int64_t kw,
                            int64_t stride, int64_t pad,
                            const int64_t *pix, int64_t npix, int64_t *acc)
{
    (void)n;
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t i = 0; i < npix; ++i) {
        int64_t b = pix[3 * i], oy = pix[3 * i + 1], ox = pix[3 * i + 2];
        for (int64_t o = 0; o < co; ++o) {
            int64_t s = 0;
            for (int64_t ky = 0; ky < kh; ++ky) {
                int64_t iy = oy * stride + ky - pad;
                if (iy < 0 || iy >= h) continue;
                for (int64_t kx = 0; kx < kw; ++kx) {
                    int64_t ix = ox * stride + kx - pad;
                    if (ix < 0 || ix >= w) continue;
                    const int8_t *xp = x + ((b * h + iy) * w + ix) * c;
                    const int8_t *wp = wt + ((o * kh + ky) * kw + kx) * c;
                    for (int64_t ci = 0; ci < c; ++ci)
                        s += (int64_t)xp[ci] * (int64_t)wp[ci];
                }
            }
            acc[i * co + o] = s;
        }
    }
}
