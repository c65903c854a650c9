/*
 * cci_oracle.c -- plain, slow, fp64 CPU oracle for layers with cross-channel
 * intragroup (CCI) sparsity (Yu et al., "Cross-Channel Intragroup Sparsity
 * Neural Network", arXiv 1910.11971).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent statement of what the
 * GPU library must compute.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it.  It shares no code, header, table or
 * helper with the CUDA library, and the CUDA library never calls it.
 *
 * Every routine is the plain definition written out: fp64 arithmetic, one
 * output at a time, reduction in ascending order of the reduction index.
 * OpenMP (when available) only splits the independent outputs across threads,
 * so results do not depend on the thread count.
 *
 * Notation (paper -> here):
 *   W (M x N), H = W x X            -> W[Cout][R], Y[n][co] (Y is H transposed)
 *   group size G, s nonzeros/group  -> G, K
 *   compressed value / index        -> values[Cout/G][R][K], idx[Cout/G][R][K]
 *   R = Cin*KH*KW, r = (kh*KW + kw)*Cin + ci for convolutions.
 *
 * Status codes mirror the library's numbering so tests can compare them:
 *   0 ok, 2 bad shape, 3 bad (G, K) or Cout % G != 0, 6 NaN in a pack input.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_SHAPE 2
#define OR_GROUP 3
#define OR_VALUE 6

static int check_group(int64_t Cout, int G, int K)
{
    if (G < 1 || G > 256 || K < 1 || K > G) return OR_GROUP;
    if (Cout <= 0 || Cout % G != 0) return OR_GROUP;
    return OR_OK;
}

int oracle_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/*
 * Pruning selection, Sec. 5.1 ("sort weights of low absolute magnitude for
 * pruning") applied under the group constraint of Sec. 3.1: for every group gi
 * of G neighbouring output channels and every input feature r, the G weights
 * W[gi*G + j][r] are ordered by decreasing |w|, equal magnitudes by increasing j
 * (the tie rule), and the first K are kept.  The kept pairs are written in
 * increasing j: values[gi][r][s] = W[gi*G + j_s][r], idx[gi][r][s] = j_s.
 * |w| of -0.0 and +0.0 are equal; +-inf is the largest magnitude; NaN is
 * rejected.  Values are copied, never rounded, so the caller may pass the
 * storage-dtype values widened to double.
 */
int oracle_pack(const double *W, int64_t Cout, int64_t R, int G, int K,
                double *values, uint8_t *idx)
{
    int st = check_group(Cout, G, K);
    if (st) return st;
    if (R <= 0) return OR_SHAPE;
    for (int64_t e = 0; e < Cout * R; ++e)
        if (isnan(W[e])) return OR_VALUE;

    const int64_t ngroups = Cout / G;
    int order[256];
    int kept[256];
    for (int64_t gi = 0; gi < ngroups; ++gi) {
        for (int64_t r = 0; r < R; ++r) {
            /* insertion sort of j = 0..G-1 by decreasing |w|; it is stable, and
             * j enters in increasing order, so ties stay in increasing j. */
            for (int j = 0; j < G; ++j) {
                double a = fabs(W[(gi * G + j) * R + r]);
                int pos = j;
                while (pos > 0 && fabs(W[(gi * G + order[pos - 1]) * R + r]) < a) {
                    order[pos] = order[pos - 1];
                    --pos;
                }
                order[pos] = j;
            }
            /* the first K survive; emit them in increasing j */
            for (int s = 0; s < K; ++s) kept[s] = order[s];
            for (int s = 1; s < K; ++s) {
                int v = kept[s], p = s;
                while (p > 0 && kept[p - 1] > v) { kept[p] = kept[p - 1]; --p; }
                kept[p] = v;
            }
            for (int s = 0; s < K; ++s) {
                const int64_t o = (gi * R + r) * K + s;
                values[o] = W[(gi * G + kept[s]) * R + r];
                idx[o] = (uint8_t)kept[s];
            }
        }
    }
    return OR_OK;
}

/*
 * Decompression of the packed format back to the M x N matrix of Sec. 3.1
 * (W-hat, with the pruned entries as zeros): Wd[gi*G + idx][r] += value for
 * every slot.  mask[co][r] counts the slots that land on (co, r); entries with
 * mask 0 are structural zeros.  A repeated index inside one (group, r) is summed,
 * which is what Alg. 2 does with such an input.  Indices >= G are rejected.
 */
int oracle_decompress(const double *values, const uint8_t *idx, int64_t Cout,
                      int64_t R, int G, int K, double *Wd, int32_t *mask)
{
    int st = check_group(Cout, G, K);
    if (st) return st;
    memset(Wd, 0, sizeof(double) * (size_t)(Cout * R));
    memset(mask, 0, sizeof(int32_t) * (size_t)(Cout * R));
    const int64_t ngroups = Cout / G;
    for (int64_t gi = 0; gi < ngroups; ++gi)
        for (int64_t r = 0; r < R; ++r)
            for (int s = 0; s < K; ++s) {
                const int64_t o = (gi * R + r) * K + s;
                if (idx[o] >= G) return OR_VALUE;
                const int64_t co = gi * G + idx[o];
                Wd[co * R + r] += values[o];
                mask[co * R + r] += 1;
            }
    return OR_OK;
}

/*
 * Alg. 1 (dense matrix product) on the decompressed weights:
 *   Y[n][co] = sum_{r ascending, mask[co][r] != 0} Wd[co][r] * X[n][r]
 * and the per-output error scale S[n][co] = sum |Wd[co][r]| * |X[n][r]| over
 * the same terms.  Structural zeros are skipped, never multiplied.  X is
 * [N][R] row-major (the paper's column-major X), Y and S are [N][Cout].
 * S may be NULL.
 */
void oracle_linear(const double *X, int64_t N, int64_t R, const double *Wd,
                   const int32_t *mask, int64_t Cout, double *Y, double *S)
{
#pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        for (int64_t co = 0; co < Cout; ++co) {
            double acc = 0.0, sc = 0.0;
            for (int64_t r = 0; r < R; ++r) {
                if (!mask[co * R + r]) continue;
                acc += Wd[co * R + r] * X[n * R + r];
                sc += fabs(Wd[co * R + r]) * fabs(X[n * R + r]);
            }
            Y[n * Cout + co] = acc;
            if (S) S[n * Cout + co] = sc;
        }
    }
}

/*
 * Alg. 2 (CCI-sparse matrix product) taken literally, with the slot loop the
 * paper leaves out for s > 1: for each group i, column j, input k and slot s,
 *   H(G*i + Idx, j) += Val * X(k, j)   with (Idx, Val) = W-hat(i, k)[s].
 * Written to the same [N][Cout] layout as oracle_linear.  Used to show that the
 * sparse loop and the dense product on the decompressed matrix agree.
 */
int oracle_linear_alg2(const double *X, int64_t N, int64_t R,
                       const double *values, const uint8_t *idx, int64_t Cout,
                       int G, int K, double *Y)
{
    int st = check_group(Cout, G, K);
    if (st) return st;
    const int64_t ngroups = Cout / G;
    for (int64_t e = 0; e < N * Cout; ++e) Y[e] = 0.0;
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < N; ++j)
        for (int64_t i = 0; i < ngroups; ++i)
            for (int64_t k = 0; k < R; ++k)
                for (int s = 0; s < K; ++s) {
                    const int64_t o = (i * R + k) * K + s;
                    const int64_t row = G * i + idx[o];
                    Y[j * Cout + row] += values[o] * X[j * R + k];
                }
    return OR_OK;
}

/*
 * Direct convolution (cross-correlation, zero padding, floor output size; no
 * dilation, groups or bias) with the decompressed weights in OHWI order:
 *   Y[b][p][q][co] = sum_{kh, kw, ci} Wd[co][(kh*KW + kw)*Cin + ci]
 *                     * X[b][p*sh - ph + kh][q*sw - pw + kw][ci]
 * taps outside the image contribute nothing.  X is NHWC [B][H][W][Cin]; the
 * output positions computed are pts[0..npts) (flattened (b*P + p)*Q + q), or all
 * B*P*Q positions in order when pts is NULL.  Y and S are [npts][Cout]; S may
 * be NULL.  The sum runs over r = (kh*KW + kw)*Cin + ci in ascending order.
 */
int oracle_conv2d(const double *X, int64_t B, int64_t H, int64_t Wi, int64_t Cin,
                  const double *Wd, const int32_t *mask, int64_t Cout, int KH,
                  int KW, int sh, int sw, int ph, int pw, const int64_t *pts,
                  int64_t npts, double *Y, double *S)
{
    if (B <= 0 || H <= 0 || Wi <= 0 || Cin <= 0 || KH <= 0 || KW <= 0 || sh <= 0 ||
        sw <= 0 || ph < 0 || pw < 0)
        return OR_SHAPE;
    const int64_t P = (H + 2 * ph - KH) / sh + 1;
    const int64_t Q = (Wi + 2 * pw - KW) / sw + 1;
    if (H + 2 * ph < KH || Wi + 2 * pw < KW) return OR_SHAPE;
    const int64_t R = (int64_t)KH * KW * Cin;
    const int64_t total = pts ? npts : B * P * Q;
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < total; ++t) {
        const int64_t n = pts ? pts[t] : t;
        const int64_t b = n / (P * Q), p = (n / Q) % P, q = n % Q;
        for (int64_t co = 0; co < Cout; ++co) {
            double acc = 0.0, sc = 0.0;
            for (int kh = 0; kh < KH; ++kh) {
                const int64_t h = p * sh - ph + kh;
                if (h < 0 || h >= H) continue;
                for (int kw = 0; kw < KW; ++kw) {
                    const int64_t w = q * sw - pw + kw;
                    if (w < 0 || w >= Wi) continue;
                    for (int64_t ci = 0; ci < Cin; ++ci) {
                        const int64_t r = ((int64_t)kh * KW + kw) * Cin + ci;
                        if (!mask[co * R + r]) continue;
                        const double x = X[((b * H + h) * Wi + w) * Cin + ci];
                        acc += Wd[co * R + r] * x;
                        sc += fabs(Wd[co * R + r]) * fabs(x);
                    }
                }
            }
            Y[t * Cout + co] = acc;
            if (S) S[t * Cout + co] = sc;
        }
    }
    return OR_OK;
}
