/*
 * fp32-ordered OBS sweep: the oracle's statement of Algorithm 2 (Eq. obs_update; with
 * the GPTAQ correction P of Proposition 1 when Pt is given) with every float32 operation
 * and its order written out, so that a float32 implementation that follows the same
 * order gives the same bits.
 *
 * TEST INFRASTRUCTURE ONLY: called by the tests and the benchmark's CPU-baseline leg,
 * never by the product path. Compiled with -ffp-contract=off; division is the IEEE
 * correctly rounded '/', rounding is rintf (half to even), fused multiply-add is fmaf.
 *
 * Operation order per row (rows are independent given R):
 *   grid (per row before the sweep, or per group of `block` columns at block start):
 *     xmin = min(0, min x); xmax = max(0, max x); if both 0: xmin = -1, xmax = 1
 *     scale = (xmax - xmin) / (float)(2^b - 1);  zero = rintf(-xmin / scale)
 *   column j:   q = clamp(rintf(w / scale) + zero, 0, 2^b - 1)
 *               what = scale * (q - zero);  E = (w - what) / R_jj
 *               w_k = fmaf(-E, R_jk, w_k) for k = j+1 .. block end - 1
 *               with P:  w_k = fmaf(w, P_jk, fmaf(-E, R_jk, w_k)), w = column j's value
 *               before it was quantized
 *   after the block [i, e): for each column c >= e:
 *               acc = 0; acc = fmaf(E_k, R_kc, acc) for k = i .. e-1 (ascending)
 *               with P, continuing: acc = fmaf(-wpre_k, P_kc, acc) for k = i .. e-1
 *               w_c = w_c - acc
 * R is read from Lt = R^T (row-major, lower), R_jk = Lt[k * n + j]; P from Pt = P^T
 * (row-major, strictly lower), P_jk = Pt[k * n + j].
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static void grid(const float *x, int64_t len, int bits, float *scale, float *zero)
{
    float xmin = 0.0f, xmax = 0.0f;
    for (int64_t k = 0; k < len; ++k) {
        if (x[k] < xmin) xmin = x[k];
        if (x[k] > xmax) xmax = x[k];
    }
    if (xmin == 0.0f && xmax == 0.0f) { xmin = -1.0f; xmax = 1.0f; }
    float maxq = (float)((1 << bits) - 1);
    float s = (xmax - xmin) / maxq;
    *scale = s;
    *zero = rintf(-xmin / s);
}

/* One row of the sweep. w: the row (n floats, updated in place as the sweep goes). */
static void sweep_row(float *w, const float *Lt, const float *Pt, int64_t n, int bits, int group,
                      int block, uint8_t *codes, float *scale, float *zero, float *E, float *pre_q,
                      float *wpre)
{
    float maxq = (float)((1 << bits) - 1);
    float s = 0.0f, z = 0.0f;
    if (group == 0) {
        grid(w, n, bits, &s, &z);
        scale[0] = s;
        zero[0] = z;
    }
    for (int64_t i = 0; i < n; i += block) {
        int64_t e = i + block < n ? i + block : n;
        if (group) {
            grid(w + i, e - i, bits, &s, &z);
            scale[i / group] = s;
            zero[i / group] = z;
        }
        for (int64_t j = i; j < e; ++j) {
            float wj = w[j];
            if (pre_q) pre_q[j] = wj;
            wpre[j - i] = wj;
            float q = rintf(wj / s) + z;
            if (q < 0.0f) q = 0.0f;
            if (q > maxq) q = maxq;
            codes[j] = (uint8_t)q;
            float what = s * (q - z);
            float err = (wj - what) / Lt[j * n + j];
            E[j] = err;
            if (Pt) {
                for (int64_t k = j + 1; k < e; ++k)
                    w[k] = fmaf(wj, Pt[k * n + j], fmaf(-err, Lt[k * n + j], w[k]));
            } else {
                for (int64_t k = j + 1; k < e; ++k)
                    w[k] = fmaf(-err, Lt[k * n + j], w[k]);
            }
        }
        for (int64_t c = e; c < n; ++c) {
            float acc = 0.0f;
            for (int64_t k = i; k < e; ++k)
                acc = fmaf(E[k], Lt[c * n + k], acc);
            if (Pt)
                for (int64_t k = i; k < e; ++k)
                    acc = fmaf(-wpre[k - i], Pt[c * n + k], acc);
            w[c] = w[c] - acc;
        }
    }
}

/*
 * Sweep the rows listed in `rows` (nrows of them; NULL = rows 0..nrows-1) of W [m x n].
 * Pt = P^T (NULL: GPTQ mode, no drift correction). Outputs are indexed by position in the
 * row list: codes/E/pre_q [nrows x n], scale/zero [nrows x ngroups]. W itself is not
 * modified. Returns 0, or -1 on bad args.
 */
int kqref_sweep32(const float *W, int64_t m, int64_t n, const float *Lt, const float *Pt, int bits,
                  int group, int block, const int64_t *rows, int64_t nrows, uint8_t *codes,
                  float *scale, float *zero, float *E, float *pre_q)
{
    if (bits < 1 || bits > 8 || block < 1 || (group != 0 && group != block) || n < 1)
        return -1;
    int64_t ngroups = group ? (n + group - 1) / group : 1;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 4) reduction(| : bad)
    for (int64_t t = 0; t < nrows; ++t) {
        int64_t r = rows ? rows[t] : t;
        if (r < 0 || r >= m) { bad = 1; continue; }
        float *w = (float *)malloc((size_t)(n + block) * sizeof(float));
        if (!w) { bad = 1; continue; }
        memcpy(w, W + r * n, (size_t)n * sizeof(float));
        sweep_row(w, Lt, Pt, n, bits, group, block, codes + t * n, scale + t * ngroups,
                  zero + t * ngroups, E + t * n, pre_q ? pre_q + t * n : NULL, w + n);
        free(w);
    }
    return bad ? -1 : 0;
}
