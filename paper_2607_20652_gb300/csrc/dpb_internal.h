// dpb_internal.h -- private declarations shared by the library's translation
// units (plan builder, C-ABI layer, kernel launchers). Not installed.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

#include "../../include/dpb.h"

struct dpb_plan {
    dpb_config cfg;             // resolved: every derived field filled in
    int device = 0;             // device current at creation; tables live there
    int sms = 0;                // its multiprocessor count (0 for a host-only plan)
    int t = 0;                  // field GF(2^t)
    uint32_t poly = 0;          // p(z), bit t set
    int code_len = 0;           // k (global) or sum of k_per_level
    uint32_t m_mask = 0;        // 2^N - 1, N = bits[levels-1]
    float inv_sqrt_d = 0.f;     // fp32(1 / sqrt(d))
    std::vector<uint32_t> M;    // [d] packed seed-matrix rows
    std::vector<uint32_t> G;    // [DPB_MAX_LEVELS * DPB_MAX_CHILDREN]
    // VH[k][q][v]: bit l = parity(inv(32 q + l) AND (v << 5k)), the part of the
    // sign word of a 32-coordinate block that the high half of an index
    // contributes, per 5-bit chunk k of that half (d <= 1024 only).
    std::vector<uint32_t> VH;   // [kvh][32][32]
    int kvh = 0;                // chunks of the high half: ceil(t / 5)
    // Tensor-core encoder tables (built when mma_encode is set):
    //  FRAG[l-1][m][chunk][lane][4]: the generator signs gamma_j of level l
    //    over 32-coordinate block m, as bf16 +-1 pairs in mma.sync B-fragment
    //    order (chunk 0: pairs 0 and 1 of the block, chunk 1: pairs 2 and 3);
    //  DD[l-1][kDedupSlots]: open-addressing table of the differences
    //    g_j ^ g_j' (j != j') of level l below 2^bits[l-1], one word per
    //    entry: (difference + 1) << 4 | j (0 = empty).
    bool mma_encode = false;
    std::vector<uint32_t> FRAG;
    std::vector<uint32_t> DD;
    // Per-level (tensor-core) encoder tables, built for DPB_SELECT_PER_LEVEL:
    //  GT: every level's generator signs gamma_j as bf16 +-1, per 64-coordinate
    //    chunk a [Delta_l][64] tile in the K-major core-matrix layout of
    //    tcgen05 (8 x 16-byte core matrices; element (n, kk) at byte
    //    (n / 8) 1024 + (kk / 8) 128 + (n % 8) 16 + (kk % 8) 2), where K
    //    position kk = 32 b + 2 i + h of the chunk holds coordinate
    //    32 (2 c + b) + i + 16 h; level l starts at word gt_off[l];
    //  VH2[k][q][v]: as VH, for every 32-coordinate block of d <= 2048 (built
    //    for every plan; max(2, kvh) chunks).
    std::vector<uint32_t> GT;
    std::vector<uint32_t> VH2;
    int64_t gt_off[DPB_MAX_LEVELS] = {};
    uint32_t *dM = nullptr;     // device copy of M
    uint32_t *dG = nullptr;     // device copy of G
    uint32_t *dVH = nullptr;    // device copy of VH
    uint32_t *dFRAG = nullptr;  // device copy of FRAG
    uint32_t *dDD = nullptr;    // device copy of DD
    uint32_t *dGT = nullptr;    // device copy of GT
    uint32_t *dVH2 = nullptr;   // device copy of VH2
    // Coset-generator scoring (DPB_SCORING_COSET_WHT), per level l >= 1:
    //  COSET[(l-1) * (nblk + 16) + m] = sign word of g0 over 32-coordinate
    //  block m (bit i = parity(M[32 m + i] AND g0)), then 16 words S_j with
    //  g_j = g0 ^ S_j (S_j in 0..15).
    std::vector<uint32_t> COSET;
    uint32_t *dCOSET = nullptr;
};

namespace dpb {

constexpr int kDedupSlots = 512;

__host__ __device__ inline uint32_t dedup_hash(uint32_t delta) {
    return (delta * 2654435761u) >> (32 - 9);
}

// The K-permuted coordinate of pair slot `pair` (0..3), half `half` (0..1) of
// lane quarter q4 in a 32-coordinate block: the tensor-core encoder gives the
// lane with q4 = lane % 4 the coordinates q4 + 4 j (j < 8), paired (j, j + 4).
__host__ __device__ inline int frag_coord(int q4, int pair, int half) { return q4 + 4 * (pair + 4 * half); }

// Builds the tensor-core encoder tables when the plan qualifies (dpb_plan.cu).
void build_mma_tables(dpb_plan *p);

// Per-level encoder (dpb_encode_pl.cu): support check, tables, launch.
dpb_status check_per_level(const dpb_config &c);
void build_per_level_tables(dpb_plan *p);
size_t encode_pl_smem(const dpb_plan *p);
cudaError_t launch_encode_pl(const dpb_plan *p, const void *x, int64_t T, const float *mu, const float *sigma,
                             const float2 *tab, int32_t *idx, float *val, float *xnorm, int32_t *status,
                             cudaStream_t stream);

// Launch shape of the tensor-core encoder: the most warps per block (16, 12,
// 8 or 4) whose shared memory fits, or 0 if none does; and that memory.
int encode_mma_warps(const dpb_plan *p);
size_t encode_mma_smem(const dpb_plan *p, int warps);
constexpr size_t kMaxSmemPerBlock = 227 * 1024;

// Lets kernel `func` use `bytes` of dynamic shared memory on the current
// device. The attribute is set the first time a kernel needs more than its
// default (and again only when a later launch needs more), so repeated
// launches make no driver call; returns the error of a failed set.
cudaError_t allow_smem(const void *func, size_t bytes);

// The warps per block (1..max_warps) that put the most warps of kernel
// `func` on an SM of the current device, by the occupancy calculator, when a
// block of w warps takes per_block + w per_warp bytes of dynamic shared
// memory (ties go to more warps per block); 0 if none fits. Cached per
// (kernel, device, sizes).
int best_warps(const void *func, int max_warps, size_t per_block, size_t per_warp);

// Records a message for dpb_last_error() and returns `s`.
dpb_status fail(dpb_status s, const char *fmt, ...);

// Builds field, seed matrix and generators on the host (dpb_plan.cu).
dpb_status resolve_and_build(const dpb_config *in, const uint32_t *generators, dpb_plan *p);

// Kernel launchers (return cudaGetLastError() of the launch).
cudaError_t launch_encode_mma(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                              const float *sigma, const float2 *tab, int32_t *idx, float *val, float *xnorm,
                              int32_t *status, cudaStream_t stream);
// tab_scratch (nullable, tab_bytes(p) bytes): where the standardisation tables
// are packed as (mu, 1 / sigma) pairs before the encoder runs.
cudaError_t launch_encode(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                          const float *sigma, int32_t *idx, float *val, float *xnorm,
                          int32_t *status, float2 *tab_scratch, cudaStream_t stream);

// Workspace: the status word (kStatusBytes, required) and, after it, the
// optional packed standardisation tables (8 bytes per feature, for 2^N up to
// 2^26; 0 bytes beyond).
constexpr size_t kStatusBytes = 256;
inline size_t tab_bytes(const dpb_plan *p) {
    const uint64_t m = (uint64_t)p->m_mask + 1;
    return m <= (1ull << 26) ? (size_t)((8 * m + 255) / 256 * 256) : 0;
}
cudaError_t launch_decode(const dpb_plan *p, const int32_t *idx, const float *val, int64_t T,
                          const float *xnorm, void *y, float *r_out, int32_t *status, cudaStream_t stream);
cudaError_t launch_backward(const dpb_plan *p, const void *x, const int32_t *idx,
                            const float *val, int64_t T, const float *sigma, const float *r_in,
                            const void *grad_y, void *grad_x, float *grad_val, int32_t *status,
                            cudaStream_t stream);

// Standardisation moments (dpb_stats.cu): whether the sampled search fits
// (kept sets of at most 64, shared memory), and the two launches.
bool stats_supported(const dpb_plan *p, size_t *smem_out);
cudaError_t launch_stats_accumulate(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                                    const float *sigma, const int32_t *sample, int32_t n_sample, double *acc,
                                    int32_t *status, cudaStream_t stream);
cudaError_t launch_stats_update(const dpb_plan *p, double *acc, float alpha, float *mu, float *sigma,
                                cudaStream_t stream);

// Dynamic shared memory (bytes) the encode kernel needs per warp / per block
// header, used both to pick the launch shape and to reject plans that do not fit.
size_t encode_smem_per_warp(const dpb_plan *p);
size_t encode_smem_header(const dpb_plan *p);

}  // namespace dpb
