/*
 * Exhaustive search over every integer code vector of one weight row.
 * Test infrastructure for the fp64 oracle (brute-force pin); not product code.
 *
 * With a diagonal Fisher the layer-level surrogate of Eq. (fisher_loss) splits
 * into independent rows, and for row i with fixed grid (scale, zero) it is
 *     L_i(q) = (1/2) F_ii * delta(q)^T Hbar delta(q),
 *     delta_k(q) = scale * (q_k - zero) - w0_k ,  q_k in {0, ..., levels-1}.
 * realq_brute_row_min enumerates all levels^n code vectors (n <= 10) with an
 * incremental evaluation of the quadratic form (one more fixed coordinate per
 * recursion level) and returns the minimum of delta^T Hbar delta and its
 * argmin.  realq_brute_row_eval evaluates the same quadratic form directly at
 * one code vector.  Both are plain C with fp64 arithmetic.
 */
#include <stdint.h>

#define MAXN 10
#define MAXLV 16

typedef struct {
    int n, levels;
    const double *H;     /* n x n, row-major */
    const double *dv;    /* n x levels: delta_k for code c at dv[k*levels + c] */
    double best;
    int cur[MAXN];
    int arg[MAXN];
} search_t;

/* s[l] = sum_{i<k} H[l][i] delta_i for l >= k; part = quadratic form over i,j < k */
static void descend(search_t *S, int k, const double *s, double part)
{
    const int n = S->n, lv = S->levels;
    const double *H = S->H;
    const double hkk = H[k * n + k];
    if (k == n - 1) {
        for (int c = 0; c < lv; ++c) {
            double d = S->dv[k * lv + c];
            double L = part + 2.0 * d * s[k] + hkk * d * d;
            if (L < S->best) {
                S->best = L;
                for (int i = 0; i < k; ++i) S->arg[i] = S->cur[i];
                S->arg[k] = c;
            }
        }
        return;
    }
    double s2[MAXN];
    for (int c = 0; c < lv; ++c) {
        double d = S->dv[k * lv + c];
        double L = part + 2.0 * d * s[k] + hkk * d * d;
        for (int l = k + 1; l < n; ++l) s2[l] = s[l] + H[l * n + k] * d;
        S->cur[k] = c;
        descend(S, k + 1, s2, L);
    }
}

double realq_brute_row_min(int n, int levels, const double *H, const double *dv, int32_t *argmin)
{
    if (n < 1 || n > MAXN || levels < 1 || levels > MAXLV) return -1.0;
    search_t S;
    S.n = n; S.levels = levels; S.H = H; S.dv = dv; S.best = 1e300;
    double s0[MAXN];
    for (int l = 0; l < n; ++l) s0[l] = 0.0;
    descend(&S, 0, s0, 0.0);
    for (int i = 0; i < n; ++i) argmin[i] = S.arg[i];
    return S.best;
}

double realq_brute_row_eval(int n, int levels, const double *H, const double *dv, const int32_t *codes)
{
    double L = 0.0;
    for (int i = 0; i < n; ++i) {
        double di = dv[i * levels + codes[i]];
        for (int j = 0; j < n; ++j) L += di * H[i * n + j] * dv[j * levels + codes[j]];
    }
    return L;
}
