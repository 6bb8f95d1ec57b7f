/*
 * dpb.h -- C ABI of the GB300 Deep Parity Bottleneck (DPB) library.
 *
 * The Deep Parity Bottleneck of "Scaling Interpretable Transformers with
 * Parity Bottleneck Layers" (arxiv 2607.20652) maps each token x in R^d to a
 * sparse code over m = 2^N features and back:
 *
 *   encode    hierarchical beam search over the parity-hashed feature
 *             hierarchy (§2.2): level 0 scores the d basis coordinates,
 *             level l scores the children p ^ g_j of the previous level's
 *             beam through the factorised inner product of Eq. 6, and the
 *             code is the top k of every candidate seen.
 *   decode    x_hat = sum_e val_e * phi_{idx_e} (§2.1), with each
 *             coordinate of phi_i generated on chip from the parity of
 *             M[iota] AND i (App. A.4, Eq. 26-27), then rescaled to |x|
 *             ("Normalized Reconstruction", §2.2).
 *   backward  gradients with respect to x and to the coefficients, through
 *             the selected features only (the selection held fixed).
 *
 * Conventions for every call:
 *   - All device pointers are plain CUDA device (or managed) pointers on the
 *     device that was current when the plan was created; host pointers are
 *     marked "host". Nothing is retained after a call returns.
 *   - Layouts are dense row-major: x, y, grad_x, grad_y are [T][d] in the
 *     plan's dtype (fp32 or bf16); idx is int32 [T][k]; val and grad_val are
 *     fp32 [T][k]; xnorm is fp32 [T]; mu and sigma are fp32 [2^N].
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream). Arguments are validated on the host before any launch;
 *     a launch failure returns DPB_ERR_CUDA. The library allocates no memory
 *     in encode/decode/backward: the caller owns every buffer, including the
 *     workspace.
 *   - Device-side checks (an index outside [0, 2^N) handed to decode or
 *     backward, a sigma <= 0) never fault: the kernel skips the bad entry and
 *     sets a sticky bit in the workspace status word; read it with
 *     dpb_workspace_status().
 *   - Errors return a dpb_status; dpb_last_error() gives a message for the
 *     calling thread's last failure.
 */
#ifndef DPB_H
#define DPB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DPB_MAX_LEVELS 8
#define DPB_MAX_CHILDREN 256

typedef enum {
    DPB_OK = 0,
    DPB_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad size or config */
    DPB_ERR_UNSUPPORTED = 2,  /* valid for the method, outside this build's limits */
    DPB_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed */
    DPB_ERR_TIMEOUT = 4,      /* reserved: a bounded device wait gave up */
    DPB_ERR_NO_MEMORY = 5,    /* plan creation could not allocate its tables */
    DPB_ERR_DEVICE = 6        /* dpb_workspace_status found a device-side error bit */
} dpb_status;

typedef enum { DPB_F32 = 0, DPB_BF16 = 1 } dpb_dtype;

/* DPB_SELECT_GLOBAL: beam `beam` at every level and a final top-k over every
 * candidate visited. DPB_SELECT_PER_LEVEL: the paper's form (§2.2 and the
 * per-level table of App. G): level l keeps its top k_per_level[l], and the
 * code is every level's kept set, level by level. */
typedef enum { DPB_SELECT_GLOBAL = 0, DPB_SELECT_PER_LEVEL = 1 } dpb_select;

/* How child scores are computed (see dpb_config.scoring). */
typedef enum { DPB_SCORING_CONTRACTION = 0, DPB_SCORING_COSET_WHT = 1 } dpb_scoring;

/* Device status bits (sticky, OR-ed by kernels into the workspace word). */
#define DPB_DEV_BAD_INDEX 0x1   /* an idx outside [0, 2^N) was skipped        */
#define DPB_DEV_BAD_SIGMA 0x2   /* a sigma <= 0 or non-finite was met         */
#define DPB_DEV_SHORT_CODE 0x4  /* fewer than k distinct candidates were seen */
#define DPB_DEV_TIMEOUT 0x8     /* a bounded wait inside a kernel gave up      */

/*
 * Configuration (§2.2 and App. G). Zero-valued optional fields are derived:
 *   d           residual width (1..4096)
 *   levels      L, counting level 0 (the paper's "2L" variant has L = 2)
 *   m_bits      N, log2 of the index space; used when bits[] is all zero
 *   bits[l]     cumulative bit boundary r_l: level l holds [2^{r_{l-1}}, 2^{r_l});
 *               derived as r_0 = ceil(log2 d), r_l = r_0 + floor(l (N - r_0) / (L-1))
 *   children[l] Delta_l for l >= 1 (children scored per parent), 1..256
 *   beam        B, beam width at every level (global mode), 1..32
 *   k           code length per token (global mode), 1..256, k <= d
 *   k_per_level K_l per level (per-level mode)
 *   select_mode dpb_select
 *   norm_match  1: y = r |x| / |r| (0 when |r| = 0); 0: y = r
 *   dtype       dpb_dtype of x, y, grad_x, grad_y
 *   field_t     t of GF(2^t); 0 = max(ceil(log2 d), ceil(r_{L-1} / 2))
 *   field_poly  p(z) as a bit mask with bit t set; 0 = z^10+z^3+1 (t = 10)
 *               and z^11+z^2+1 (t = 11) as in App. A.4 Eq. 24, otherwise the
 *               smallest irreducible trinomial, else pentanomial
 *   generator_seed  seed of the generator draw (splitmix64, see the plan)
 *   scoring     DPB_SCORING_CONTRACTION: child scores by the dense
 *               contraction of Eq. 6 (any generators). DPB_SCORING_COSET_WHT:
 *               a variant outside the paper, for generators given by the
 *               caller where every level's 16 generators are one coset
 *               g0 ^ {0, ..., 15} of the span of index bits 0..3: a parent's 16
 *               child scores are then a 16-point Walsh-Hadamard transform of
 *               16 bucket sums of x (.) phi~_{p ^ g0} (bucket = iota mod 16).
 *               Global selection, bf16, beam <= 8, d a multiple of 32 up to 1024.
 */
typedef struct dpb_config {
    int32_t d;
    int32_t levels;
    int32_t m_bits;
    int32_t bits[DPB_MAX_LEVELS];
    int32_t children[DPB_MAX_LEVELS];
    int32_t beam;
    int32_t k;
    int32_t k_per_level[DPB_MAX_LEVELS];
    int32_t select_mode;
    int32_t norm_match;
    int32_t dtype;
    int32_t field_t;
    uint32_t field_poly;
    uint64_t generator_seed;
    int32_t scoring;
    int32_t reserved;             /* 0 */
} dpb_config;

typedef struct dpb_plan dpb_plan;

/*
 * dpb_plan_create -- validate `cfg`, build the field GF(2^t), the seed matrix
 * M (App. A.4 Eq. 22: row iota = coord(xi_iota) | coord(xi_iota^{-1}) << t,
 * with inverses xi^{2^t-2}, Eq. 25) and the generators of every level (§2.2:
 * g_j < 2^{r_l} with a set bit at or above r_{l-1}), and upload them to the
 * current device. `generators` (host, nullable) overrides the draw: it holds
 * DPB_MAX_LEVELS rows of DPB_MAX_CHILDREN words, row l = g_0..g_{Delta_l - 1}
 * of the transition l-1 -> l (row 0 ignored); each must obey the level rule.
 * Without it, level l draws splitmix64 (Steele, Lea, Flood 2014) from state
 * generator_seed ^ (l * 0x9E3779B97F4A7C15), takes the top r_l bits and keeps
 * new valid values. On success *out owns a plan; free it with
 * dpb_plan_destroy. On a host with no CUDA device the plan is host-only:
 * dpb_plan_config / dpb_plan_tables / dpb_code_length work and every compute
 * call returns DPB_ERR_CUDA. Errors: INVALID_ARG (bad config), UNSUPPORTED
 * (outside the limits above), NO_MEMORY / CUDA (table upload).
 */
dpb_status dpb_plan_create(const dpb_config *cfg, const uint32_t *generators, dpb_plan **out);

/* Free a plan and its device tables (no-op on NULL). The caller must make
 * sure no call using the plan is still running on the device. */
dpb_status dpb_plan_destroy(dpb_plan *plan);

/* Copy the resolved configuration (every derived field filled in) to host *out. */
dpb_status dpb_plan_config(const dpb_plan *plan, dpb_config *out);

/* Copy the plan's tables to host memory: M_out[d] (packed seed-matrix rows,
 * nullable) and G_out[DPB_MAX_LEVELS * DPB_MAX_CHILDREN] (generators, row l as
 * above, unused entries 0; nullable). */
dpb_status dpb_plan_tables(const dpb_plan *plan, uint32_t *M_out, uint32_t *G_out);

/* Code length per token: k (global mode) or sum_l k_per_level[l]. */
dpb_status dpb_code_length(const dpb_plan *plan, int32_t *k_out);

/* Bytes of workspace for T tokens (256-byte aligned pointer required): 256
 * bytes for the device status word, then 8 * 2^N bytes (for 2^N <= 2^26)
 * where dpb_encode packs the standardisation tables as (mu, 1 / sigma) pairs,
 * so that each candidate costs one table load instead of two. Any workspace of
 * at least 256 bytes is accepted; a smaller one than this size only leaves the
 * tables unpacked (same results, slower with tables). The status word must be
 * zero-filled once before its first use; the workspace may be reused by every
 * call on the same stream. Calls that run concurrently need separate
 * workspaces. */
dpb_status dpb_workspace_size(const dpb_plan *plan, int64_t T, size_t *bytes);

/*
 * dpb_encode -- §2.2 encoder for T tokens (T = 0 is a no-op).
 *   x      [T][d] plan dtype, 16-byte aligned
 *   mu, sigma  [2^N] fp32 standardisation tables (§2.2 "Score
 *          Standardization": z = (s - mu_i) / sigma_i); both NULL = identity
 *   idx    out int32 [T][k]; val out fp32 [T][k] (signed z): each row sorted
 *          by (|val| descending, idx ascending)
 *   xnorm  out fp32 [T] = |x_t| (nullable)
 * Level 0 scores are x_i; level l >= 1 scores are <gamma_j, phi~_p (.) x>
 * accumulated in fp32 (Eq. 6). Errors: INVALID_ARG, CUDA.
 */
dpb_status dpb_encode(const dpb_plan *plan, const void *x, int64_t T, const float *mu,
                      const float *sigma, int32_t *idx, float *val, float *xnorm,
                      void *workspace, size_t workspace_bytes, void *stream);

/*
 * dpb_decode -- §2.1 decoder: r_t = sum_e val[t][e] * phi_{idx[t][e]} with
 * phi_i = e_i for i < d (Eq. 2) and generated parity signs / sqrt(d)
 * otherwise (Eq. 1, 26, 27), accumulated in fp32; y_t = r_t * xnorm_t / |r_t|
 * when the plan has norm_match (y_t = 0 if |r_t| = 0), else y_t = r_t.
 *   idx, val  [T][k] (any order; k = dpb_code_length); entries outside
 *             [0, 2^N) are skipped and flagged DPB_DEV_BAD_INDEX
 *   xnorm     [T] fp32, required iff norm_match
 *   y         out [T][d] plan dtype, 16-byte aligned
 *   r_out     out fp32 [T][d], 16-byte aligned, nullable: r_t itself, kept
 *             for dpb_backward (which then does not rebuild it)
 */
dpb_status dpb_decode(const dpb_plan *plan, const int32_t *idx, const float *val, int64_t T,
                      const float *xnorm, void *y, float *r_out, void *workspace,
                      size_t workspace_bytes, void *stream);

/*
 * dpb_backward -- gradients of L(decode(encode(x))) with the selected set
 * held fixed. With g = grad_y, r and y as in dpb_decode, c = |x| / |r|:
 *   dL/dr      = c (g - (<g,r>/|r|^2) r)   (norm_match)   or g
 *   grad_val_e = <phi_e, dL/dr>
 *   grad_x     = sum_e (grad_val_e / sigma_e) phi_e + (<g,r>/|r|) x / |x|
 * (the last term only with norm_match; zero gradients when |r| = 0).
 *   x, grad_y  [T][d] plan dtype; idx, val [T][k]; sigma [2^N] fp32 nullable
 *   r          fp32 [T][d], 16-byte aligned, nullable: the r_out of the
 *              dpb_decode of this code; given, it replaces the rebuilding of
 *              r (same value up to fp32 summation order)
 *   grad_x     out [T][d] plan dtype; grad_val out fp32 [T][k]
 */
dpb_status dpb_backward(const dpb_plan *plan, const void *x, const int32_t *idx,
                        const float *val, int64_t T, const float *sigma, const float *r,
                        const void *grad_y, void *grad_x, float *grad_val, void *workspace,
                        size_t workspace_bytes, void *stream);

/*
 * dpb_stats_accumulate -- moment sums of the score standardisation (§2.2
 * "Score Standardization": each feature's score is standardised by EMAs of
 * its mean and deviation, taken over the tokens on which it is a candidate;
 * levels >= 1 take them on a 64-token sub-sample of the batch). Adds to acc,
 * fp64 [3][2^N] = count, sum of s, sum of s^2 per feature, where s is the raw
 * (unstandardised) score:
 *   level 0    every row of x: each basis coordinate i < d adds s = x_t[i];
 *   level >= 1 the rows sample[0..n_sample) only: the encoder's search is run
 *              again on each (kept set of a level = its top beam, or top
 *              k_per_level[l] in per-level mode, by |z| under mu/sigma), and
 *              every distinct child p ^ g_j it scores at a level l >= 1 adds
 *              s = <phi_c, x_t> (accumulated in fp32).
 *   x          [T][d] plan dtype, 16-byte aligned
 *   mu, sigma  the tables the encoder selects with (both NULL = identity)
 *   sample     device int32 [n_sample] row numbers in [0, T); a row may
 *              repeat; a row outside [0, T) is skipped and flagged
 *              DPB_DEV_BAD_INDEX (NULL allowed when n_sample = 0)
 *   acc        device fp64 [3][2^N] (24 * 2^N bytes, 8-byte aligned, owned by
 *              the caller), zero before a batch's first call; sums are fp64
 *              atomics, so their last bits depend on the order of arrival
 * The search rounds like the encoder but not in the same order: where two
 * scores sit within fp32 rounding of each other at a kept-set cut, the
 * candidates counted here can differ from those the encoder visited.
 * Errors: INVALID_ARG, UNSUPPORTED (a kept set above 64), CUDA.
 */
dpb_status dpb_stats_accumulate(const dpb_plan *plan, const void *x, int64_t T, const float *mu,
                                const float *sigma, const int32_t *sample, int32_t n_sample,
                                double *acc, void *workspace, size_t workspace_bytes, void *stream);

/*
 * dpb_stats_update -- one EMA step of the standardisation tables from acc,
 * then acc = 0. For each feature with n = count >= 1: m = sum / n and
 * mu += alpha (m - mu); with n >= 2 also v = sqrt(max(sum s^2 / n - m^2, 0))
 * (the population deviation) and sigma += alpha (v - sigma); features with
 * n = 0 keep their moments. With 0 < alpha < 1 a positive sigma stays
 * positive. mu, sigma: device fp32 [2^N], updated in place (fp64 arithmetic,
 * rounded to fp32). Data-parallel callers sum acc across ranks (one
 * all-reduce) before this call; every rank then makes the same update.
 * Errors: INVALID_ARG (alpha outside (0, 1), NULL or misaligned buffers), CUDA.
 */
dpb_status dpb_stats_update(const dpb_plan *plan, double *acc, float alpha, float *mu, float *sigma,
                            void *stream);

/*
 * dpb_forward -- the layer's forward pass: the §2.2 encoder (dpb_encode) and
 * then the §2.1 decoder with on-chip signs (Eq. 1-2, App. A.4 Eq. 26-27;
 * dpb_decode) over the same T rows, as two kernels on `stream`.
 *   x, mu, sigma, idx, val, xnorm  as in dpb_encode (device; idx/val [T, k]
 *                                  are written, as the backward needs them;
 *                                  xnorm [T] is required with norm_match)
 *   y                              [T, d] in the plan's dtype (device, out)
 *   r_out                          optional fp32 [T, d] r before norm matching
 *                                  (device, out; NULL to skip), as in dpb_decode
 * The caller owns every buffer; the workspace is that of dpb_encode.
 * Errors: those of either call (the decode is not launched when the encode
 * fails).
 */
dpb_status dpb_forward(const dpb_plan *plan, const void *x, int64_t T, const float *mu, const float *sigma,
                       int32_t *idx, float *val, float *xnorm, void *y, float *r_out, void *workspace,
                       size_t workspace_bytes, void *stream);

/* Read (and with clear != 0, zero) the workspace status word: synchronises
 * `stream`, writes the sticky DPB_DEV_* bits to host *status_out, and returns
 * DPB_ERR_DEVICE if any bit is set, else DPB_OK. */
dpb_status dpb_workspace_status(const void *workspace, int clear, int32_t *status_out,
                                void *stream);

/*
 * dpb_encode_noalloc -- dpb_encode for callers that cannot allocate device
 * memory. The paper has no counterpart: this is a deployment convenience.
 * Some callers cannot call cudaMalloc or hand over a workspace, for example a
 * plug-in that runs inside another runtime which owns every device
 * allocation and passes it only its input and output buffers. This entry
 * point takes the same inputs and outputs as dpb_encode but no workspace: its
 * scratch (the device status word) lives in a file-scope device array of
 * 4096 bytes that every GPU which loads the library keeps until the process
 * exits. It allocates nothing: no cudaMalloc, no cudaFree, no allocating
 * library routine.
 *   status_out  device int32 (nullable): receives the DPB_DEV_* bits of this
 *               call (the scratch word is cleared at the start of each call)
 * The status word is all the scratch this call needs, for every plan and
 * every T, so no plan is rejected for its size: the packed (mu, 1/sigma)
 * table copy that dpb_encode keeps in a workspace of dpb_workspace_size
 * bytes is not made here, and a standardised call reads mu and sigma from
 * the two caller tables instead (same results, one more load per candidate,
 * so slower with tables). The first call on a device looks up the
 * array's device address (cudaGetSymbolAddress); make that first call before
 * any stream capture. Every call on a device shares the one array, so calls
 * whose kernels overlap on the GPU (different streams, or several host
 * threads) race on it and must be serialised by the caller.
 */
dpb_status dpb_encode_noalloc(const dpb_plan *plan, const void *x, int64_t T, const float *mu,
                              const float *sigma, int32_t *idx, float *val, float *xnorm,
                              int32_t *status_out, void *stream);

/*
 * dpb_debug_set_wait_limit -- test hook for the bounded waits of the
 * per-level (tcgen05) encoder; the paper has no counterpart. Every
 * mbarrier wait of that kernel's main loop (a generator-tile copy landing,
 * the MMAs of a chunk or level finishing) gives up after `tries` polls for
 * the launches that follow, from any thread; -1 restores the default
 * (2^20 polls). A wait that gives up stops the block: the kernel sets
 * DPB_DEV_TIMEOUT in the workspace status, waits (with the default bound)
 * for its copies and MMAs still in flight, frees its tensor memory and
 * returns; that call's codes are incomplete. With tries = 0 every such wait
 * gives up at once, which lets a test exercise that path without a fault.
 * Returns DPB_ERR_INVALID_ARG for tries < -1.
 */
dpb_status dpb_debug_set_wait_limit(int32_t tries);

/* Static description of a status code. */
const char *dpb_status_string(dpb_status s);

/* Message describing the calling thread's last failed call ("" if none). */
const char *dpb_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* DPB_H */
