/*
 * dpb_oracle.c -- plain CPU oracle of the Deep Parity Bottleneck (DPB).
 *
 * TEST INFRASTRUCTURE. Only the tests, the smoke check and the CPU-baseline
 * leg of the benchmark may load this file. The product library never links,
 * loads or calls it, and it shares no code, header, table or constant
 * generator with the CUDA path.
 *
 * Every quantity is computed in double precision, straight from the
 * definitions in "Scaling Interpretable Transformers with Parity Bottleneck
 * Layers" (arxiv 2607.20652), slowly and without blocking or fusion:
 *
 *   field GF(2^t)           App. A.2 (polynomial basis, Eq. 10 and 11)
 *   seed matrix M           App. A.4, Eq. 22 and 25
 *   hashed direction        §2.1 Eq. 1, App. A.4 Eq. 26 and 27
 *   basis override          §2.1 Eq. 2
 *   generators / children   §2.2 (child map, Eq. 5)
 *   encoder (beam search)   §2.2 (level-by-level scoring, AbsTopK)
 *   standardisation         §2.2 "Score Standardization"
 *   decoder                 §2.1 (x_hat = sum_i a_i phi_i)
 *   normalised output       §2.2 "Normalized Reconstruction"
 *   backward                not written in the paper; derived by the chain
 *                           rule with the selected set held fixed
 *
 * Readings of the paper that this file takes where the paper is silent or
 * inconsistent (listed with their reasons in the design notes):
 *   R1  d need not be 2^t: the field is GF(2^t) with t >= ceil(log2 d) and
 *       rows 0..d-1 of the construction are used, scaled by 1/sqrt(d).
 *   R3  bits(i): the low t bits are the half that meets coord(xi), the high
 *       t bits the half that meets coord(xi^{-1}).
 *   R4  indices are 0-based: indices 0..d-1 are the basis directions.
 *   R6  the generators of the transition l-1 -> l lie below 2^{r_l} and have
 *       a set bit at or above r_{l-1}; level l's children are scored at l.
 *   R7  generators come from splitmix64 (Steele, Lea, Flood 2014) with state
 *       seed ^ (l * 0x9E3779B97F4A7C15), by rejection (new, valid values).
 *   R8  the candidates of a level form a set: each index is scored once.
 *   R9  ordering is (|z| descending, index ascending) everywhere.
 *   R10 global selection: beam B at every level, final code = top k over
 *       every candidate visited (all d basis entries and every level's set).
 *   R12 normalised output: y = r * |x| / |r|, and y = 0 when |r| = 0.
 *   R16 a feature is "considered" on a token when the search scores it
 *       there: every basis coordinate on every token (level 0), every
 *       distinct child of the previous level's kept set (level >= 1).
 *   R17 the EMA step: with n considered occurrences in the sample, mean
 *       m = (sum s) / n and population deviation v = sqrt(sum s^2 / n - m^2);
 *       mu += alpha (m - mu) when n >= 1, sigma += alpha (v - sigma) when
 *       n >= 2; untouched features keep their moments.
 *   R18 level 0 takes every token of the batch, levels >= 1 a caller-given
 *       list of token rows (the paper's 64-token sub-sample).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_MAX_LEVELS 8

/* ------------------------------------------------------------------ */
/* GF(2) polynomials and the field GF(2^t)  (App. A.2)                 */
/* ------------------------------------------------------------------ */

/* Degree of a binary polynomial (bit j = coefficient of z^j); -1 for 0. */
static int poly_degree(uint64_t p)
{
    int d = -1;
    while (p) {
        d++;
        p >>= 1;
    }
    return d;
}

/* Remainder of a divided by b over GF(2) (schoolbook long division). */
static uint64_t poly_mod(uint64_t a, uint64_t b)
{
    int db = poly_degree(b);
    int da = poly_degree(a);
    while (da >= db) {
        a ^= b << (da - db);
        da = poly_degree(a);
    }
    return a;
}

/* 1 if poly (degree t, bit t set) has no factor of degree 1..t/2.
 * App. A.2: p(z) must be irreducible for GF(2^t) to be a field. */
int orc_poly_is_irreducible(int t, uint32_t poly)
{
    if (t < 1 || poly_degree(poly) != t)
        return 0;
    for (uint64_t f = 2; poly_degree(f) <= t / 2; f++) {
        if (poly_degree(f) < 1)
            continue;
        if (poly_mod(poly, f) == 0)
            return 0;
    }
    return 1;
}

/* Product in GF(2^t): carry-less multiplication, then reduction mod p(z)
 * (App. A.2: "multiplied as polynomials and the result is reduced"). */
uint32_t orc_gf_mul(uint32_t a, uint32_t b, int t, uint32_t poly)
{
    uint64_t prod = 0;
    for (int j = 0; j < t; j++)
        if ((b >> j) & 1u)
            prod ^= (uint64_t)a << j;
    return (uint32_t)poly_mod(prod, poly);
}

/* xi^{-1} = xi^{2^t - 2} by repeated multiplication (App. A.4, Eq. 25),
 * with the convention 0^{-1} = 0 (App. A.3). */
uint32_t orc_gf_inv(uint32_t a, int t, uint32_t poly)
{
    if (a == 0)
        return 0;
    uint64_t e = ((uint64_t)1 << t) - 2;
    uint32_t r = 1;
    for (uint64_t n = 0; n < e; n++)
        r = orc_gf_mul(r, a, t, poly);
    return r;
}

/* Absolute trace Tr(y) = y + y^2 + y^4 + ... + y^{2^{t-1}} (App. A.2, Eq. 11).
 * Returned as the field element; Lemma A.2 says it is 0 or 1. */
uint32_t orc_gf_trace(uint32_t y, int t, uint32_t poly)
{
    uint32_t s = 0, p = y;
    for (int j = 0; j < t; j++) {
        s ^= p;
        p = orc_gf_mul(p, p, t, poly);
    }
    return s;
}

/* Kloosterman codeword bit c_{a,b}(xi) = Tr(a xi + b xi^{-1}) (App. A.3, Eq. 12). */
uint32_t orc_kloosterman_bit(uint32_t a, uint32_t b, uint32_t xi, int t, uint32_t poly)
{
    uint32_t v = orc_gf_mul(a, xi, t, poly) ^ orc_gf_mul(b, orc_gf_inv(xi, t, poly), t, poly);
    return orc_gf_trace(v, t, poly);
}

/* ------------------------------------------------------------------ */
/* Seed matrix and directions  (§2.1 Eq. 1-2, App. A.4 Eq. 22, 26, 27)  */
/* ------------------------------------------------------------------ */

/* Row iota of M packed in one word: coord(xi_iota) in the low t bits and
 * coord(xi_iota^{-1}) in the next t bits (App. A.4, Eq. 22; reading R3). */
void orc_seed_matrix(int d, int t, uint32_t poly, uint32_t *M)
{
    for (int iota = 0; iota < d; iota++)
        M[iota] = (uint32_t)iota | (orc_gf_inv((uint32_t)iota, t, poly) << t);
}

/* Parity of the number of set bits of v (the compiler's bit-count builtin). */
static int bit_parity(uint32_t v)
{
    return __builtin_parity(v);
}

/* Sign (+1 or -1) of coordinate iota of the hashed direction of index i:
 * R(M bits(i))_iota with R(0) = +1, R(1) = -1 (App. A.4, Eq. 26 and 27). */
static double hashed_sign(const uint32_t *M, uint32_t i, int iota)
{
    return bit_parity(M[iota] & i) ? -1.0 : 1.0;
}

/* phi_i as a dense vector of length d: e_i for i < d (Eq. 2, reading R4),
 * otherwise R(M bits(i)) / sqrt(d) (Eq. 1). */
void orc_phi(int d, const uint32_t *M, uint32_t i, double *out)
{
    if (i < (uint32_t)d) {
        for (int iota = 0; iota < d; iota++)
            out[iota] = (iota == (int)i) ? 1.0 : 0.0;
        return;
    }
    double s = 1.0 / sqrt((double)d);
    for (int iota = 0; iota < d; iota++)
        out[iota] = s * hashed_sign(M, i, iota);
}

/* The hashed direction of any index, without the basis override (Eq. 1). */
void orc_phi_tilde(int d, const uint32_t *M, uint32_t i, double *out)
{
    double s = 1.0 / sqrt((double)d);
    for (int iota = 0; iota < d; iota++)
        out[iota] = s * hashed_sign(M, i, iota);
}

/* ------------------------------------------------------------------ */
/* Generators of the hierarchy  (§2.2; readings R6, R7)                 */
/* ------------------------------------------------------------------ */

/* splitmix64 (Steele, Lea, Flood, OOPSLA 2014): one step of the generator. */
static uint64_t splitmix64_next(uint64_t *state)
{
    uint64_t z = (*state += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* G[l * gstride + j] = g_j of the transition l-1 -> l, for l = 1..levels-1.
 * Draw g uniformly below 2^{r_l}; keep it if it has a set bit at or above
 * r_{l-1} (so the child lies in level l) and is not already kept.
 * Returns 0, or -1 if a level asks for more generators than exist. */
int orc_generators(int levels, const int *bits, const int *children, uint64_t seed,
                   uint32_t *G, int gstride)
{
    for (int l = 1; l < levels; l++) {
        uint64_t available = ((uint64_t)1 << bits[l]) - ((uint64_t)1 << bits[l - 1]);
        if (children[l] < 1 || (uint64_t)children[l] > available || children[l] > gstride)
            return -1;
        uint64_t state = seed ^ ((uint64_t)l * 0x9E3779B97F4A7C15ULL);
        int n = 0;
        while (n < children[l]) {
            uint32_t g = (uint32_t)(splitmix64_next(&state) >> (64 - bits[l]));
            if ((g >> bits[l - 1]) == 0)
                continue;
            int seen = 0;
            for (int m = 0; m < n; m++)
                if (G[l * gstride + m] == g)
                    seen = 1;
            if (seen)
                continue;
            G[l * gstride + n] = g;
            n++;
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Encoder  (§2.2)                                                     */
/* ------------------------------------------------------------------ */

typedef struct {
    uint32_t idx;
    double z;
    int exact; /* score is a plain coordinate read (level 0, no tables) */
} cand_t;

/* Order of reading R9: |z| descending, then index ascending. */
static int cand_cmp(const void *pa, const void *pb)
{
    const cand_t *a = (const cand_t *)pa, *b = (const cand_t *)pb;
    double za = fabs(a->z), zb = fabs(b->z);
    if (za > zb)
        return -1;
    if (za < zb)
        return 1;
    return (a->idx < b->idx) ? -1 : (a->idx > b->idx) ? 1 : 0;
}

/* Relative gap at a cut of n sorted candidates keeping the first `keep`:
 * the smallest (|z_a| - |z_b|) / |z_a| over a kept a and a dropped b of which
 * at least one has an inexact score. Two level-0 scores read without tables
 * are the same number on every implementation, so a tie between them is
 * settled by index everywhere and is not a near-tie. */
static double cut_gap(const cand_t *sorted, int n, int keep)
{
    if (keep >= n || keep <= 0)
        return INFINITY;
    int last_inexact_kept = -1, first_inexact_dropped = -1;
    for (int e = 0; e < keep; e++)
        if (!sorted[e].exact)
            last_inexact_kept = e;
    for (int e = keep; e < n && first_inexact_dropped < 0; e++)
        if (!sorted[e].exact)
            first_inexact_dropped = e;
    double gap = INFINITY;
    if (last_inexact_kept >= 0) {
        double a = fabs(sorted[last_inexact_kept].z), b = fabs(sorted[keep].z);
        double g = a > 0.0 ? (a - b) / a : 0.0;
        if (g < gap)
            gap = g;
    }
    if (first_inexact_dropped >= 0) {
        double a = fabs(sorted[keep - 1].z), b = fabs(sorted[first_inexact_dropped].z);
        double g = a > 0.0 ? (a - b) / a : 0.0;
        if (g < gap)
            gap = g;
    }
    return gap;
}

/* Score of index c against x by the direct inner product <phi_c, x>.
 * (The GPU uses the factorised form of Eq. 6; the oracle deliberately does not.) */
static double direct_score(int d, const uint32_t *M, uint32_t c, const double *x)
{
    if (c < (uint32_t)d)
        return x[c];
    double s = 0.0;
    for (int iota = 0; iota < d; iota++)
        s += hashed_sign(M, c, iota) * x[iota];
    return s / sqrt((double)d);
}

/* z = (s - mu_c) / sigma_c; absent tables mean mu = 0, sigma = 1. */
static double standardise(double s, uint32_t c, const double *mu, const double *sigma)
{
    double m = mu ? mu[c] : 0.0;
    double sd = sigma ? sigma[c] : 1.0;
    return (s - m) / sd;
}

/*
 * Global-mode encoder (reading R10). For each token t (row x[t*d .. t*d+d)):
 *   level 0: every basis index i < d is a candidate with score x_i;
 *            the beam is the top `beam` of them.
 *   level l: the candidates are the distinct children p ^ g_j of the
 *            previous beam, each scored by a direct inner product; the
 *            beam becomes the top `beam` of this level.
 *   code:    the top k of every candidate seen, in the order of R9,
 *            val = signed standardised score.
 * xnorm[t] = |x_t| (may be NULL). mingap[t] = smallest relative gap at any
 * cut (beam cuts and the final cut), used to flag near-ties (may be NULL).
 * Returns 0, -1 on bad arguments, -2 if k exceeds the candidates seen.
 */
int orc_encode(int d, int levels, const int *bits, const int *children, int beam, int k,
               const uint32_t *M, const uint32_t *G, int gstride,
               const double *x, long T, const double *mu, const double *sigma,
               int32_t *idx, double *val, double *xnorm, double *mingap)
{
    (void)bits;
    if (d < 1 || levels < 1 || levels > ORC_MAX_LEVELS || beam < 1 || k < 1)
        return -1;
    long cap = d;
    for (int l = 1; l < levels; l++)
        cap += (long)beam * children[l];
    cand_t *all = (cand_t *)malloc(sizeof(cand_t) * cap);
    cand_t *lvl = (cand_t *)malloc(sizeof(cand_t) * cap);
    uint32_t *parents = (uint32_t *)malloc(sizeof(uint32_t) * (size_t)(beam > d ? beam : d));
    if (!all || !lvl || !parents) {
        free(all);
        free(lvl);
        free(parents);
        return -1;
    }
    int rc = 0;
    for (long t = 0; t < T && rc == 0; t++) {
        const double *xt = x + t * d;
        double gap = INFINITY;
        int nall = 0;

        /* level 0: every basis coordinate; its score is a coordinate read */
        int nl = 0;
        for (int i = 0; i < d; i++) {
            lvl[nl].idx = (uint32_t)i;
            lvl[nl].z = standardise(xt[i], (uint32_t)i, mu, sigma);
            lvl[nl].exact = (mu == NULL && sigma == NULL);
            nl++;
        }
        for (int l = 0;; l++) {
            memcpy(all + nall, lvl, sizeof(cand_t) * (size_t)nl);
            nall += nl;
            if (l == levels - 1)
                break;
            /* beam of level l: its top `beam` candidates */
            qsort(lvl, (size_t)nl, sizeof(cand_t), cand_cmp);
            int nb = nl < beam ? nl : beam;
            double g = cut_gap(lvl, nl, nb);
            if (g < gap)
                gap = g;
            for (int b = 0; b < nb; b++)
                parents[b] = lvl[b].idx;
            /* level l+1: the distinct children p ^ g_j of the beam (R8) */
            nl = 0;
            for (int b = 0; b < nb; b++) {
                for (int j = 0; j < children[l + 1]; j++) {
                    uint32_t c = parents[b] ^ G[(l + 1) * gstride + j];
                    int seen = 0;
                    for (int m = 0; m < nl; m++)
                        if (lvl[m].idx == c)
                            seen = 1;
                    if (!seen) {
                        lvl[nl].idx = c;
                        lvl[nl].exact = 0;
                        nl++;
                    }
                }
            }
            for (int m = 0; m < nl; m++)
                lvl[m].z = standardise(direct_score(d, M, lvl[m].idx, xt), lvl[m].idx, mu, sigma);
        }
        if (k > nall) {
            rc = -2;
            break;
        }
        /* the code: top k of every candidate seen */
        qsort(all, (size_t)nall, sizeof(cand_t), cand_cmp);
        double g = cut_gap(all, nall, k);
        if (g < gap)
            gap = g;
        for (int e = 0; e < k; e++) {
            idx[t * k + e] = (int32_t)all[e].idx;
            val[t * k + e] = all[e].z;
        }
        if (xnorm) {
            double s = 0.0;
            for (int i = 0; i < d; i++)
                s += xt[i] * xt[i];
            xnorm[t] = sqrt(s);
        }
        if (mingap)
            mingap[t] = gap;
    }
    free(all);
    free(lvl);
    free(parents);
    return rc;
}

/*
 * Per-level encoder in the paper's own form (§2.2 and the per-level
 * configuration table of App. G): level 0 keeps its top K_0 basis entries;
 * level l scores the distinct children of level l-1's kept set and keeps its
 * top K_l. The code is every level's kept set, level by level, each in the
 * order of R9. Output rows have sum_l K_l entries. Returns 0 or -1.
 */
int orc_encode_per_level(int d, int levels, const int *children, const int *k_per_level,
                         const uint32_t *M, const uint32_t *G, int gstride,
                         const double *x, long T, const double *mu, const double *sigma,
                         int32_t *idx, double *val, double *mingap)
{
    if (d < 1 || levels < 1 || levels > ORC_MAX_LEVELS)
        return -1;
    int ktot = 0, cap = d;
    for (int l = 0; l < levels; l++) {
        if (k_per_level[l] < 1)
            return -1;
        ktot += k_per_level[l];
        if (l >= 1 && k_per_level[l - 1] * children[l] > cap)
            cap = k_per_level[l - 1] * children[l];
    }
    cand_t *lvl = (cand_t *)malloc(sizeof(cand_t) * (size_t)cap);
    uint32_t *parents = (uint32_t *)malloc(sizeof(uint32_t) * (size_t)cap);
    if (!lvl || !parents) {
        free(lvl);
        free(parents);
        return -1;
    }
    int rc = 0;
    for (long t = 0; t < T && rc == 0; t++) {
        const double *xt = x + t * d;
        double gap = INFINITY;
        int out = 0, nl = 0;
        for (int i = 0; i < d; i++) {
            lvl[nl].idx = (uint32_t)i;
            lvl[nl].z = standardise(xt[i], (uint32_t)i, mu, sigma);
            lvl[nl].exact = (mu == NULL && sigma == NULL);
            nl++;
        }
        for (int l = 0;; l++) {
            qsort(lvl, (size_t)nl, sizeof(cand_t), cand_cmp);
            if (k_per_level[l] > nl) {
                rc = -1;
                break;
            }
            double g = cut_gap(lvl, nl, k_per_level[l]);
            if (g < gap)
                gap = g;
            for (int e = 0; e < k_per_level[l]; e++) {
                idx[t * ktot + out] = (int32_t)lvl[e].idx;
                val[t * ktot + out] = lvl[e].z;
                parents[e] = lvl[e].idx;
                out++;
            }
            if (l == levels - 1)
                break;
            int np = k_per_level[l];
            nl = 0;
            for (int b = 0; b < np; b++) {
                for (int j = 0; j < children[l + 1]; j++) {
                    uint32_t c = parents[b] ^ G[(l + 1) * gstride + j];
                    int seen = 0;
                    for (int m = 0; m < nl; m++)
                        if (lvl[m].idx == c)
                            seen = 1;
                    if (!seen) {
                        lvl[nl].idx = c;
                        lvl[nl].exact = 0;
                        nl++;
                    }
                }
            }
            for (int m = 0; m < nl; m++)
                lvl[m].z = standardise(direct_score(d, M, lvl[m].idx, xt), lvl[m].idx, mu, sigma);
        }
        if (mingap)
            mingap[t] = gap;
    }
    free(lvl);
    free(parents);
    return rc;
}

/* ------------------------------------------------------------------ */
/* Standardisation moments  (§2.2 "Score Standardization"; R16-R18)     */
/* ------------------------------------------------------------------ */

/*
 * Adds the moment sums of the raw scores s to acc, three arrays of m doubles
 * (count, sum of s, sum of s^2), over the occurrences where a feature is a
 * candidate (R16, R18):
 *   level 0    every basis coordinate i < d on every token t < T: s = x_t[i];
 *   level l>0  on each sampled token only: every distinct child p ^ g_j of the
 *              previous level's kept set, s = <phi_c, x_t>.
 * The kept set of a level is its top keep[l] candidates by standardised score
 * (R9 order; mu/sigma as in the encoder, both NULL = identity), so the search
 * is the encoder's: keep[l] = beam (global mode) or K_l (per-level mode).
 * Returns 0, or -1 on bad arguments (a sampled row outside [0, T)).
 */
int orc_stats_accumulate(int d, int levels, const int *children, const int *keep,
                         const uint32_t *M, const uint32_t *G, int gstride,
                         const double *x, long T, const double *mu, const double *sigma,
                         const int32_t *sample, int n_sample, double *acc, long m)
{
    if (d < 1 || levels < 1 || levels > ORC_MAX_LEVELS || m < d || n_sample < 0)
        return -1;
    for (int s = 0; s < n_sample; s++)
        if (sample[s] < 0 || sample[s] >= T)
            return -1;
    double *cnt = acc, *sum = acc + m, *sq = acc + 2 * m;

    /* level 0: every token considers every basis coordinate */
    for (long t = 0; t < T; t++)
        for (int i = 0; i < d; i++) {
            double v = x[t * d + i];
            cnt[i] += 1.0;
            sum[i] += v;
            sq[i] += v * v;
        }

    long cap = d;
    for (int l = 1; l < levels; l++)
        if ((long)keep[l - 1] * children[l] > cap)
            cap = (long)keep[l - 1] * children[l];
    cand_t *lvl = (cand_t *)malloc(sizeof(cand_t) * (size_t)cap);
    double *raw = (double *)malloc(sizeof(double) * (size_t)cap);
    uint32_t *parents = (uint32_t *)malloc(sizeof(uint32_t) * (size_t)cap);
    if (!lvl || !raw || !parents) {
        free(lvl);
        free(raw);
        free(parents);
        return -1;
    }
    for (int s = 0; s < n_sample; s++) {
        const double *xt = x + (long)sample[s] * d;
        int nl = 0;
        for (int i = 0; i < d; i++) {
            lvl[nl].idx = (uint32_t)i;
            lvl[nl].z = standardise(xt[i], (uint32_t)i, mu, sigma);
            lvl[nl].exact = 0;
            nl++;
        }
        for (int l = 1; l < levels; l++) {
            /* kept set of level l-1 */
            qsort(lvl, (size_t)nl, sizeof(cand_t), cand_cmp);
            int np = nl < keep[l - 1] ? nl : keep[l - 1];
            for (int b = 0; b < np; b++)
                parents[b] = lvl[b].idx;
            /* the distinct children of the kept set (R8) */
            nl = 0;
            for (int b = 0; b < np; b++) {
                for (int j = 0; j < children[l]; j++) {
                    uint32_t c = parents[b] ^ G[l * gstride + j];
                    int seen = 0;
                    for (int q = 0; q < nl; q++)
                        if (lvl[q].idx == c)
                            seen = 1;
                    if (!seen) {
                        lvl[nl].idx = c;
                        lvl[nl].exact = 0;
                        nl++;
                    }
                }
            }
            /* each is considered once on this token: its raw score joins the sums */
            for (int q = 0; q < nl; q++) {
                uint32_t c = lvl[q].idx;
                raw[q] = direct_score(d, M, c, xt);
                if ((long)c < m) {
                    cnt[c] += 1.0;
                    sum[c] += raw[q];
                    sq[c] += raw[q] * raw[q];
                }
                lvl[q].z = standardise(raw[q], c, mu, sigma);
            }
        }
    }
    free(lvl);
    free(raw);
    free(parents);
    return 0;
}

/*
 * One EMA step of the standardisation tables from the sums of
 * orc_stats_accumulate (R17), then acc = 0. For feature i with n = acc
 * count >= 1: m = sum / n, mu_i += alpha (m - mu_i); with n >= 2 also
 * v = sqrt(max(sum s^2 / n - m^2, 0)), sigma_i += alpha (v - sigma_i).
 */
void orc_stats_update(long m, double *acc, double alpha, double *mu, double *sigma)
{
    double *cnt = acc, *sum = acc + m, *sq = acc + 2 * m;
    for (long i = 0; i < m; i++) {
        double n = cnt[i];
        if (n >= 1.0) {
            double mean = sum[i] / n;
            mu[i] += alpha * (mean - mu[i]);
            if (n >= 2.0) {
                double var = sq[i] / n - mean * mean;
                double v = sqrt(var > 0.0 ? var : 0.0);
                sigma[i] += alpha * (v - sigma[i]);
            }
        }
        cnt[i] = sum[i] = sq[i] = 0.0;
    }
}

/* ------------------------------------------------------------------ */
/* Decoder  (§2.1, "Normalized Reconstruction" in §2.2)                 */
/* ------------------------------------------------------------------ */

/* r = sum_e val_e * phi_{idx_e} for one token (length d). */
static void reconstruct(int d, const uint32_t *M, const int32_t *idx, const double *val, int k,
                        double *r, double *phi)
{
    for (int i = 0; i < d; i++)
        r[i] = 0.0;
    for (int e = 0; e < k; e++) {
        orc_phi(d, M, (uint32_t)idx[e], phi);
        for (int i = 0; i < d; i++)
            r[i] += val[e] * phi[i];
    }
}

static double norm2(const double *v, int d)
{
    double s = 0.0;
    for (int i = 0; i < d; i++)
        s += v[i] * v[i];
    return sqrt(s);
}

/* y_t = r_t, or r_t * xnorm_t / |r_t| when norm_match (y = 0 if |r_t| = 0). */
int orc_decode(int d, int k, int norm_match, const uint32_t *M,
               const int32_t *idx, const double *val, long T, const double *xnorm, double *y)
{
    double *phi = (double *)malloc(sizeof(double) * (size_t)d);
    if (!phi)
        return -1;
    for (long t = 0; t < T; t++) {
        double *yt = y + t * d;
        reconstruct(d, M, idx + t * k, val + t * k, k, yt, phi);
        if (norm_match) {
            double nr = norm2(yt, d);
            double c = nr > 0.0 ? xnorm[t] / nr : 0.0;
            for (int i = 0; i < d; i++)
                yt[i] = nr > 0.0 ? yt[i] * c : 0.0;
        }
    }
    free(phi);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Backward of decode(encode(x)) with the selected set held fixed       */
/* ------------------------------------------------------------------ */

/*
 * val_e = (<phi_e, x> - mu_e) / sigma_e, r = sum_e val_e phi_e and, when
 * norm_match, y = |x| r / |r|. With g = dL/dy:
 *   dL/dr   = c (g - (<g,r>/|r|^2) r),  c = |x|/|r|      (norm_match)
 *           = g                                           (otherwise)
 *   grad_val_e = <phi_e, dL/dr>
 *   grad_x     = sum_e (grad_val_e / sigma_e) phi_e  +  (<g,r>/|r|) x/|x|
 * where the last term (through |x|) is present only with norm_match.
 * |r| = 0 gives zero gradients (y = 0 there); |x| = 0 drops the last term.
 */
int orc_backward(int d, int k, int norm_match, const uint32_t *M,
                 const double *x, const int32_t *idx, const double *val, long T,
                 const double *sigma, const double *gy, double *gx, double *gval)
{
    double *phi = (double *)malloc(sizeof(double) * (size_t)d);
    double *r = (double *)malloc(sizeof(double) * (size_t)d);
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    if (!phi || !r || !h) {
        free(phi);
        free(r);
        free(h);
        return -1;
    }
    for (long t = 0; t < T; t++) {
        const double *xt = x + t * d, *gt = gy + t * d;
        const int32_t *it = idx + t * k;
        const double *vt = val + t * k;
        double *gxt = gx + t * d, *gvt = gval + t * k;
        double direct = 0.0, nx = norm2(xt, d);
        if (norm_match) {
            reconstruct(d, M, it, vt, k, r, phi);
            double nr = norm2(r, d);
            if (nr > 0.0) {
                double gr = 0.0;
                for (int i = 0; i < d; i++)
                    gr += gt[i] * r[i];
                double c = nx / nr;
                for (int i = 0; i < d; i++)
                    h[i] = c * (gt[i] - (gr / (nr * nr)) * r[i]);
                direct = nx > 0.0 ? gr / nr : 0.0;
            } else {
                for (int i = 0; i < d; i++)
                    h[i] = 0.0;
            }
        } else {
            for (int i = 0; i < d; i++)
                h[i] = gt[i];
        }
        for (int i = 0; i < d; i++)
            gxt[i] = nx > 0.0 ? direct * xt[i] / nx : 0.0;
        for (int e = 0; e < k; e++) {
            orc_phi(d, M, (uint32_t)it[e], phi);
            double s = 0.0;
            for (int i = 0; i < d; i++)
                s += phi[i] * h[i];
            gvt[e] = s;
            double sd = sigma ? sigma[it[e]] : 1.0;
            for (int i = 0; i < d; i++)
                gxt[i] += (s / sd) * phi[i];
        }
    }
    free(phi);
    free(r);
    free(h);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Whole-field tables for the tests (plain loops over the functions     */
/* above; nothing here is used by the encoder, decoder or backward)     */
/* ------------------------------------------------------------------ */

/* mul[a * 2^t + b] = a b, inv[a] = a^{-1}, tr[a] = Tr(a); any may be NULL. */
void orc_gf_tables(int t, uint32_t poly, uint32_t *mul, uint32_t *inv, uint32_t *tr)
{
    uint32_t q = 1u << t;
    for (uint32_t a = 0; a < q; a++) {
        if (inv)
            inv[a] = orc_gf_inv(a, t, poly);
        if (tr)
            tr[a] = orc_gf_trace(a, t, poly);
        if (mul)
            for (uint32_t b = 0; b < q; b++)
                mul[(size_t)a * q + b] = orc_gf_mul(a, b, t, poly);
    }
}
