/* Exhaustive nearest-codeword search over the implicit linear-constrained
 * codebook {A z + B : z in {0,1,2,3}^d} (Sec. 2.1 Eq. vq_assign applied to
 * the codebook of Sec. 2.2 Eq. lc_codebook).
 *
 * TEST INFRASTRUCTURE ONLY: part of the CPU oracle. It enumerates all 4^d
 * codewords for every weight group; it is only meant for tiny matrices.
 *
 * W is m x n row-major fp64; group g of row r is W[r, g*d .. g*d+d-1].
 * A is d x d row-major (codeword_j = sum_k A[j][k] z_k + B[j]).
 * Ties keep the first codeword in enumeration order (z_0 fastest).
 * Returns 0 on success, -1 on bad arguments.
 */
#include <stdint.h>
#include <stdlib.h>

int lcvq_oracle_brute_nearest(const double *W, int64_t m, int64_t n, int d,
                              const double *A, const double *B,
                              uint8_t *codes, double *dist)
{
    if (d < 1 || d > 10 || n % d != 0 || m < 0)
        return -1;
    const int64_t G = n / d;
    const int64_t K = (int64_t)1 << (2 * d);
    double *cb = (double *)malloc(sizeof(double) * (size_t)(K * d));
    if (!cb)
        return -1;
    /* Materialise the codebook once: codeword index k holds digit z_j = (k >> 2j) & 3. */
    for (int64_t k = 0; k < K; ++k) {
        for (int j = 0; j < d; ++j) {
            double acc = B[j];
            for (int i = 0; i < d; ++i)
                acc += A[j * d + i] * (double)((k >> (2 * i)) & 3);
            cb[k * d + j] = acc;
        }
    }
    for (int64_t r = 0; r < m; ++r) {
        for (int64_t g = 0; g < G; ++g) {
            const double *w = W + r * n + g * d;
            double best = -1.0;
            int64_t arg = 0;
            for (int64_t k = 0; k < K; ++k) {
                double e = 0.0;
                for (int j = 0; j < d; ++j) {
                    double t = w[j] - cb[k * d + j];
                    e += t * t;
                }
                if (best < 0.0 || e < best) {
                    best = e;
                    arg = k;
                }
            }
            for (int j = 0; j < d; ++j)
                codes[r * n + g * d + j] = (uint8_t)((arg >> (2 * j)) & 3);
            dist[r * G + g] = best;
        }
    }
    free(cb);
    return 0;
}
