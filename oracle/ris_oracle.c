/*
 * ris_oracle.c -- plain, slow, fp64 CPU oracle for RIS prefill sparse attention.
 *
 * TEST INFRASTRUCTURE. Only the tests, the smoke check and the benchmark's CPU
 * baseline leg load this file's library. The product path (the CUDA library) never
 * calls it and shares no code with it.
 *
 * What it computes, each piece written from the method's definition:
 *   - Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As Easy as
 *     1, 2, 3", SC'11): the counter-based generator that draws the sampled pairs.
 *   - The Stochastic and Structural mask definitions (paper, Methods, "Sampling Modes:
 *     Stochastic and Structural"), the streaming OR of all seeds into one master mask
 *     (Methods, "Memory-Bounded Geometry Generation") and the per-seed masks.
 *   - RoPE with linear or YaRN position extension (Methods, "Dynamic RoPE Scaling";
 *     Results, "RoPE Scaling: Linear versus YaRN"; YaRN per Peng et al. 2023).
 *   - Masked softmax attention with one softmax over the whole selected key set
 *     (Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax (PFUS)").
 *
 * Readings taken where the paper is silent (each listed in the design notes):
 *   - a pair (i, j<i) is kept by seed s iff a 32-bit Philox word is below
 *     thr(p) = min(2^32, floor(p * 2^32 + 0.5)); the word is number (j mod 4) of
 *     Philox4x32-10 with key (seed, head_key) and counter (j/4, i, stream, layer_key),
 *     stream 0 for Stochastic draws and 1 for Structural global draws;
 *   - Structural: K = floor(d*N + 0.5) (the paper's B_max), B = max(1, min(floor(N/10), K)),
 *     blocks start at 0, each block is a causal clique, d_clique = C / N^2 with C the
 *     number of causal clique pairs, d_global = max(0, d - d_clique);
 *   - the forced set of row i is the local window {i-W < j <= i} plus the anchors
 *     {j < A}; W >= 1 keeps the diagonal so no row is empty;
 *   - density 1 (or the dense mode) is every causal pair j <= i;
 *   - the index-draw sampler (the paper's torch.randint wording, Methods, "Memory-Bounded
 *     Geometry Generation") replaces the per-pair Bernoulli test of the random part: row i
 *     of seed s draws K indices with replacement, draw t being j_t = floor(u_t * N / 2^32)
 *     with u_t word (t mod 4) of Philox4x32-10 with key (seed, head_key) and counter
 *     (t/4, i, stream + 2, layer_key); draws with j_t < i are kept (causal filter) and
 *     repeats merge (set semantics). K = floor(d N + 0.5) for Stochastic and
 *     floor(d_global N + 0.5) for the Structural global part.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------- */
/* Philox4x32-10 (SC'11, the 4x32 member with 10 rounds).                      */
/* ------------------------------------------------------------------------- */
#define PHILOX_M0 0xD2511F53u /* multiplier applied to counter word 0 */
#define PHILOX_M1 0xCD9E8D57u /* multiplier applied to counter word 2 */
#define PHILOX_W0 0x9E3779B9u /* Weyl key increment, key word 0 */
#define PHILOX_W1 0xBB67AE85u /* Weyl key increment, key word 1 */

/* One Philox round: two 32x32->64 products, the high halves xored with the other
 * counter words and the round key, the low halves passed through. */
static void philox_round(uint32_t c[4], const uint32_t k[2])
{
    uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)c[0];
    uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)c[2];
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c[1] ^ k[0];
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c[3] ^ k[1];
    uint32_t n3 = lo0;
    c[0] = n0;
    c[1] = n1;
    c[2] = n2;
    c[3] = n3;
}

void ora_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
    uint32_t k[2] = {key[0], key[1]};
    for (int r = 0; r < 10; ++r) {
        philox_round(c, k);
        k[0] += PHILOX_W0; /* the key is bumped between rounds */
        k[1] += PHILOX_W1;
    }
    out[0] = c[0];
    out[1] = c[1];
    out[2] = c[2];
    out[3] = c[3];
}

/* n independent evaluations: ctr[n][4], key[n][2] -> out[n][4]. */
void ora_philox_batch(int64_t n, const uint32_t *ctr, const uint32_t *key, uint32_t *out)
{
    for (int64_t t = 0; t < n; ++t)
        ora_philox4x32_10(ctr + 4 * t, key + 2 * t, out + 4 * t);
}

/* ------------------------------------------------------------------------- */
/* Sampling parameters.                                                        */
/* ------------------------------------------------------------------------- */

/* Bernoulli threshold on a uniform 32-bit word: keep iff word < thr(p). */
uint64_t ora_threshold(double p)
{
    if (!(p > 0.0)) return 0;
    double t = floor(p * 4294967296.0 + 0.5);
    if (t >= 4294967296.0) return (uint64_t)1 << 32;
    return (uint64_t)t;
}

/* Structural Mode block geometry (Methods, "Sampling Modes"): block size
 * B = min(0.1 N, B_max) with B_max = round(d N) (the B_max column of the sub-1%
 * sweet-spot table pins round(d N) at N = 65536), and the clique cost deducted from the
 * global allowance: d_eff = d_clique + d_global. */
void ora_structural(int64_t N, double d, int64_t *K_out, int64_t *B_out, int64_t *C_out,
                    double *d_clique_out, double *d_global_out)
{
    int64_t K = (int64_t)floor(d * (double)N + 0.5);
    int64_t tenth = N / 10;
    int64_t B = K < tenth ? K : tenth;
    if (B < 1) B = 1;
    int64_t nb = N / B;
    int64_t r = N - nb * B;
    int64_t C = nb * (B * (B + 1) / 2) + r * (r + 1) / 2;
    double d_clique = (double)C / ((double)N * (double)N);
    double d_global = d - d_clique;
    if (d_global < 0.0) d_global = 0.0;
    *K_out = K;
    *B_out = B;
    *C_out = C;
    *d_clique_out = d_clique;
    *d_global_out = d_global;
}

/* Mask specification; mirrored by a ctypes Structure in oracle/__init__.py. */
typedef struct {
    int64_t N;
    int32_t mode; /* 0 Stochastic, 1 Structural, 2 Dense */
    int32_t n_seeds;
    double density;
    const uint32_t *seeds;
    int32_t seed_index;   /* -1: union over all seeds; s >= 0: seed s alone */
    int32_t local_window; /* W >= 1 */
    int32_t n_anchor;     /* A >= 0 */
    uint32_t head_key;
    uint32_t layer_key;
    int32_t sampler; /* 0: Bernoulli test per causal pair; 1: index draws with replacement */
} ora_mask_spec;

typedef struct {
    int dense;
    uint32_t stream;
    uint64_t thr;
    int64_t B;     /* Structural block size, 0 for Stochastic */
    int64_t draws; /* index draws per row and seed (sampler 1) */
} mask_derived;

static mask_derived derive(const ora_mask_spec *m)
{
    mask_derived x;
    memset(&x, 0, sizeof(x));
    x.dense = (m->mode == 2) || (m->density >= 1.0);
    if (m->mode == 1) {
        int64_t K, B, C;
        double dc, dg;
        ora_structural(m->N, m->density, &K, &B, &C, &dc, &dg);
        x.B = B;
        x.stream = 1;
        x.thr = ora_threshold(dg);
        x.draws = (int64_t)floor(dg * (double)m->N + 0.5);
    } else {
        x.B = 0;
        x.stream = 0;
        x.thr = ora_threshold(m->density);
        x.draws = (int64_t)floor(m->density * (double)m->N + 0.5);
    }
    return x;
}

/* The 32-bit uniform word drawn for pair (i, j) by seed value `seed`. */
static uint32_t pair_word(const ora_mask_spec *m, const mask_derived *x, uint32_t seed,
                          int64_t i, int64_t j)
{
    uint32_t ctr[4] = {(uint32_t)(j / 4), (uint32_t)i, x->stream, m->layer_key};
    uint32_t key[2] = {seed, m->head_key};
    uint32_t out[4];
    ora_philox4x32_10(ctr, key, out);
    return out[j % 4];
}

/* Is the causal pair (i, j), j <= i, in the mask? Definition, term by term. */
static int keep_pair(const ora_mask_spec *m, const mask_derived *x, int64_t i, int64_t j)
{
    if (j > i) return 0;                        /* causal */
    if (x->dense) return 1;                     /* dense causal upper bound */
    if (j > i - m->local_window) return 1;      /* local window, includes the diagonal */
    if (j < m->n_anchor) return 1;              /* global anchors over the first tokens */
    if (m->mode == 1 && (i / x->B) == (j / x->B)) return 1; /* Structural block clique */
    if (m->sampler != 0) return 0; /* random part comes from the index draws */
    /* stochastic draws (Stochastic: whole budget; Structural: global remainder) */
    int s0 = m->seed_index < 0 ? 0 : m->seed_index;
    int s1 = m->seed_index < 0 ? m->n_seeds : m->seed_index + 1;
    for (int s = s0; s < s1; ++s) {
        if ((uint64_t)pair_word(m, x, m->seeds[s], i, j) < x->thr) return 1;
    }
    return 0;
}

/* Index-draw sampler: mark hit[j] = 1 for every j < i drawn for row i by the selected seeds. */
static void row_draws(const ora_mask_spec *m, const mask_derived *x, int64_t i, unsigned char *hit)
{
    int s0 = m->seed_index < 0 ? 0 : m->seed_index;
    int s1 = m->seed_index < 0 ? m->n_seeds : m->seed_index + 1;
    for (int s = s0; s < s1; ++s) {
        for (int64_t t = 0; t < x->draws; ++t) {
            uint32_t ctr[4] = {(uint32_t)(t / 4), (uint32_t)i, x->stream + 2, m->layer_key};
            uint32_t key[2] = {m->seeds[s], m->head_key};
            uint32_t out[4];
            ora_philox4x32_10(ctr, key, out);
            int64_t j = (int64_t)(((uint64_t)out[t % 4] * (uint64_t)m->N) >> 32);
            if (j < i) hit[j] = 1;
        }
    }
}

/* Membership of keys 0..i of row i: keep[j] = 1 iff (i, j) is in the mask. */
static void row_members(const ora_mask_spec *m, const mask_derived *x, int64_t i, unsigned char *keep)
{
    for (int64_t j = 0; j <= i; ++j) keep[j] = (unsigned char)keep_pair(m, x, i, j);
    if (m->sampler != 0 && !x->dense) row_draws(m, x, i, keep);
}

/* Number of kept keys of each requested row. */
void ora_mask_counts(const ora_mask_spec *m, const int64_t *rows, int64_t nrows, int64_t *counts)
{
    mask_derived x = derive(m);
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < nrows; ++r) {
        int64_t i = rows[r], c = 0;
        unsigned char *keep = (unsigned char *)malloc((size_t)i + 1);
        row_members(m, &x, i, keep);
        for (int64_t j = 0; j <= i; ++j) c += keep[j];
        free(keep);
        counts[r] = c;
    }
}

/* Kept keys of each requested row, ascending; row r writes cols[off[r] .. off[r+1]). */
void ora_mask_cols(const ora_mask_spec *m, const int64_t *rows, int64_t nrows, const int64_t *off,
                   int64_t *cols)
{
    mask_derived x = derive(m);
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < nrows; ++r) {
        int64_t i = rows[r], w = off[r];
        unsigned char *keep = (unsigned char *)malloc((size_t)i + 1);
        row_members(m, &x, i, keep);
        for (int64_t j = 0; j <= i; ++j)
            if (keep[j]) cols[w++] = j;
        free(keep);
    }
}

/* Bitmap words of each requested row: bit (j mod 32) of word (j / 32) is pair (i, j);
 * words_per_row words are written per row, bits beyond the diagonal are zero. */
void ora_mask_bits(const ora_mask_spec *m, const int64_t *rows, int64_t nrows, int64_t words_per_row,
                   uint32_t *bits)
{
    mask_derived x = derive(m);
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < nrows; ++r) {
        int64_t i = rows[r];
        uint32_t *out = bits + r * words_per_row;
        unsigned char *keep = (unsigned char *)malloc((size_t)i + 1);
        row_members(m, &x, i, keep);
        memset(out, 0, sizeof(uint32_t) * (size_t)words_per_row);
        for (int64_t j = 0; j <= i && j / 32 < words_per_row; ++j)
            if (keep[j]) out[j / 32] |= (uint32_t)1 << (j % 32);
        free(keep);
    }
}

/* ------------------------------------------------------------------------- */
/* RoPE with position extension.                                               */
/* ------------------------------------------------------------------------- */

/* Rotation frequencies f[k], k < D/2, and the magnitude scale of the rotated vectors.
 * kind: 0 none, 1 plain, 2 linear, 3 YaRN. s is the resolved extension factor.
 *   plain:  f = theta^(-2k/D)
 *   linear: f = plain / s  (positions compressed by s)
 *   YaRN:   r = L_native * plain / (2 pi); g = clamp((r - alpha)/(beta - alpha), 0, 1);
 *           f = (1 - g) * plain / s + g * plain; both q and k scaled by 0.1 ln s + 1. */
void ora_rope_freqs(int kind, double theta, int64_t native_len, double s, double alpha, double beta,
                    int D, double *f, double *mscale)
{
    const double two_pi = 6.283185307179586476925286766559;
    for (int k = 0; k < D / 2; ++k) {
        double plain = pow(theta, -2.0 * (double)k / (double)D);
        double val = plain;
        if (kind == 2) {
            val = plain / s;
        } else if (kind == 3) {
            double r = (double)native_len * plain / two_pi;
            double g = (r - alpha) / (beta - alpha);
            if (g < 0.0) g = 0.0;
            if (g > 1.0) g = 1.0;
            val = (1.0 - g) * plain / s + g * plain;
        }
        f[k] = val;
    }
    *mscale = (kind == 3) ? 0.1 * log(s) + 1.0 : 1.0;
}

/* Rotate-half RoPE in place on x[n][H][D] at positions pos[n]:
 *   x'_c     = x_c cos a - x_{c+D/2} sin a
 *   x'_{c+D/2} = x_{c+D/2} cos a + x_c sin a,   a = pos * f_c,  then times mscale. */
void ora_rope_apply(double *x, const double *pos, int64_t n, int H, int D, const double *f,
                    double mscale)
{
    int half = D / 2;
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < n; ++t) {
        for (int h = 0; h < H; ++h) {
            double *row = x + (t * H + h) * (int64_t)D;
            for (int c = 0; c < half; ++c) {
                double a = pos[t] * f[c];
                double ca = cos(a), sa = sin(a);
                double x0 = row[c], x1 = row[c + half];
                row[c] = (x0 * ca - x1 * sa) * mscale;
                row[c + half] = (x1 * ca + x0 * sa) * mscale;
            }
        }
    }
}

/* ------------------------------------------------------------------------- */
/* Masked softmax attention, one softmax over the whole selected set (PFUS).   */
/* ------------------------------------------------------------------------- */

/* For each requested row r (token rows[r]) and query head h, with g = floor(h * Hkv / Hq):
 *   z_j = <q_r,h , k_j,g> / sqrt(D)            for j in the row's key set
 *   o_r,h = sum_j softmax(z)_j v_j,g,           lse_r,h = log sum_j exp(z_j)
 * q_rows[nrows][Hq][D] holds the (already rotated) query rows, k and v are [N][Hkv][D],
 * keys of row r are cols[off[r] .. off[r+1]). */
void ora_attention(const double *q_rows, const double *k, const double *v, int64_t N, int Hq,
                   int Hkv, int D, int64_t nrows, const int64_t *off, const int64_t *cols,
                   double *out, double *lse)
{
    (void)N;
    double inv_sqrt_d = 1.0 / sqrt((double)D);
#pragma omp parallel
    {
        int64_t cap = 0;
        double *z = NULL;
#pragma omp for schedule(dynamic, 1)
        for (int64_t r = 0; r < nrows; ++r) {
            int64_t n = off[r + 1] - off[r];
            if (n > cap) {
                free(z);
                cap = n;
                z = (double *)malloc(sizeof(double) * (size_t)cap);
            }
            for (int h = 0; h < Hq; ++h) {
                int g = (int)(((int64_t)h * Hkv) / Hq);
                const double *q = q_rows + (r * Hq + h) * (int64_t)D;
                double *o = out + (r * Hq + h) * (int64_t)D;
                double zmax = -INFINITY;
                for (int64_t t = 0; t < n; ++t) {
                    const double *kj = k + (cols[off[r] + t] * Hkv + g) * (int64_t)D;
                    double acc = 0.0;
                    for (int c = 0; c < D; ++c) acc += q[c] * kj[c];
                    z[t] = acc * inv_sqrt_d;
                    if (z[t] > zmax) zmax = z[t];
                }
                double sum = 0.0;
                for (int64_t t = 0; t < n; ++t) sum += exp(z[t] - zmax);
                double l = zmax + log(sum);
                for (int c = 0; c < D; ++c) o[c] = 0.0;
                for (int64_t t = 0; t < n; ++t) {
                    double p = exp(z[t] - l);
                    const double *vj = v + (cols[off[r] + t] * Hkv + g) * (int64_t)D;
                    for (int c = 0; c < D; ++c) o[c] += p * vj[c];
                }
                if (lse) lse[r * Hq + h] = l;
            }
        }
        free(z);
    }
}

void ora_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int ora_get_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
