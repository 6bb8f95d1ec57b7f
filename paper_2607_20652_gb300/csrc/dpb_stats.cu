// Standardisation moments (§2.2 "Score Standardization"): per-feature sums of
// the raw score over the occurrences where the feature is a candidate, and the
// EMA step of the mean and deviation tables.
//
//   level 0    every token considers every basis coordinate, s = x_i: a
//              column reduction of x (HBM-bound, one pass over x).
//   level >= 1 only the sampled rows (the paper's 64-token sub-sample): one
//              block per row re-runs the encoder's search (kept set of each
//              level = its top keep[l] by standardised score, children
//              p ^ g_j, each distinct child scored once) and adds every
//              child's raw score to the sums.
//   update     a pass over the 2^N count words; only touched features read
//              their sums, move their moments and clear the sums.
#include <cuda_runtime.h>

#include <cstdint>

#include "dpb_device.cuh"
#include "dpb_internal.h"

namespace dpb {
namespace {

constexpr int kColThreads = 256;
constexpr int kColRows = 256;     // rows per block of the column pass
constexpr int kColChunk = 32;     // rows per fp32 partial before it joins the fp64 sums
constexpr int kSearchThreads = 512;
constexpr int kSearchWarps = kSearchThreads / 32;
constexpr int kMaxKeep = 64;

struct StatsArgs {
    const void *x;
    int64_t T;
    int d;
    int levels;
    int keep[DPB_MAX_LEVELS];
    int children[DPB_MAX_LEVELS];
    const uint32_t *M;
    const uint32_t *G;  // [DPB_MAX_LEVELS][DPB_MAX_CHILDREN]
    const float *mu, *sigma;
    const int32_t *sample;
    double *acc;        // [3][m]
    int64_t m;
    float inv_sqrt_d;
    int cap;            // per-level candidate slots (smem)
    int32_t *status;
};

__device__ __forceinline__ void add_moments(double *acc, int64_t m, uint32_t c, double s, double n = 1.0) {
    atomicAdd(acc + c, n);
    atomicAdd(acc + m + c, s);
    atomicAdd(acc + 2 * m + c, s * s);
}

// ---- level 0: column sums of x --------------------------------------------------

template <typename Tio>
__global__ void __launch_bounds__(kColThreads) stats_columns_kernel(const Tio *x, int64_t T, int d,
                                                                    double *acc, int64_t m) {
    const int col = blockIdx.y * kColThreads + threadIdx.x;
    if (col >= d) return;
    const int64_t r0 = (int64_t)blockIdx.x * kColRows;
    const int64_t r1 = r0 + kColRows < T ? r0 + kColRows : T;
    double s = 0.0, q = 0.0;
    for (int64_t r = r0; r < r1; r += kColChunk) {
        const int64_t re = r + kColChunk < r1 ? r + kColChunk : r1;
        float fs = 0.f, fq = 0.f;
#pragma unroll 8
        for (int64_t i = r; i < re; ++i) {
            const float v = ld_elem(x, i * d + col);
            fs += v;
            fq = fmaf(v, v, fq);
        }
        s += fs;
        q += fq;
    }
    atomicAdd(acc + m + col, s);
    atomicAdd(acc + 2 * m + col, q);
    if (blockIdx.x == 0) atomicAdd(acc + col, (double)T);
}

// ---- levels >= 1: the search on the sampled rows ---------------------------------

// The encoder's standardisation, with the same fp32 arithmetic.
__device__ __forceinline__ float z_of(float s, uint32_t c, const StatsArgs &a) {
    return a.mu ? zscore(s, c, a.mu, a.sigma, nullptr, a.status) : s;
}

// Ordering priority of a candidate (R9 order: larger first): |z| bits, then
// the complement of the index. Distinct indices give distinct priorities.
__device__ __forceinline__ uint64_t prio(float z, uint32_t c) {
    return ((uint64_t)akey(z) << 32) | (uint64_t)(~c);
}

// Block-wide sum of one value per thread (every thread gets the total).
__device__ __forceinline__ int block_sum(int v, int *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    __syncthreads();  // red is free again
    if (lane == 0) red[warp] = v;
    __syncthreads();
    int t = 0;
#pragma unroll
    for (int w = 0; w < kSearchWarps; ++w) t += red[w];
    return t;
}

// The keep largest priorities among n slots (slots with zb < 0 are not
// candidates): writes their indices to par and returns how many. PR(i) gives
// slot i's priority. The threshold is the keep-th largest priority, built bit
// by bit from the top (priorities are distinct).
template <typename PR>
__device__ int select_top(int n, int keep, const float *zb, PR pr, uint32_t *par, int *red, int *cnt,
                          const uint32_t *cid) {
    int valid = 0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) valid += zb[i] >= 0.f;
    valid = block_sum(valid, red);
    const int K = keep < valid ? keep : valid;
    uint64_t tau = 0;
    if (K < valid) {
        for (int bit = 63; bit >= 0; --bit) {
            const uint64_t cand = tau | (1ull << bit);
            int c = 0;
            for (int i = threadIdx.x; i < n; i += blockDim.x)
                if (zb[i] >= 0.f && pr(i) >= cand) ++c;
            if (block_sum(c, red) >= K) tau = cand;
        }
    }
    if (threadIdx.x == 0) *cnt = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x)
        if (zb[i] >= 0.f && pr(i) >= tau) par[atomicAdd(cnt, 1)] = cid[i];
    __syncthreads();
    return K;
}

template <typename Tio>
__global__ void __launch_bounds__(kSearchThreads, 1) stats_search_kernel(StatsArgs a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int d = a.d;
    float *xs = reinterpret_cast<float *>(smem);          // [d]
    uint32_t *Ms = smem + d;                             // [d]
    uint32_t *par = Ms + d;                              // [kMaxKeep]
    uint32_t *gen = par + kMaxKeep;                      // [DPB_MAX_CHILDREN]
    uint32_t *gsort = gen + DPB_MAX_CHILDREN;            // [DPB_MAX_CHILDREN] ascending
    int *red = reinterpret_cast<int *>(gsort + DPB_MAX_CHILDREN);  // [kSearchWarps + 1]
    float *zb = reinterpret_cast<float *>(red + kSearchWarps + 4);  // [cap] |z| (-1: not a candidate)
    uint32_t *cid = reinterpret_cast<uint32_t *>(zb + a.cap);       // [cap] candidate index

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int32_t row = a.sample[blockIdx.x];
    if (row < 0 || row >= a.T) {
        if (threadIdx.x == 0) set_status(a.status, DPB_DEV_BAD_INDEX);
        return;
    }
    const Tio *xr = static_cast<const Tio *>(a.x) + (int64_t)row * d;
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        xs[i] = ld_elem(xr, i);
        Ms[i] = a.M[i];
    }
    __syncthreads();
    // level 0: the basis coordinates
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        zb[i] = fabsf(z_of(xs[i], (uint32_t)i, a));
        cid[i] = (uint32_t)i;
    }
    __syncthreads();
    int np = select_top(
        d, a.keep[0], zb, [&](int i) { return prio(zb[i], cid[i]); }, par, red, red + kSearchWarps, cid);

    for (int l = 1; l < a.levels; ++l) {
        const int nch = a.children[l];
        for (int j = threadIdx.x; j < nch; j += blockDim.x) gen[j] = a.G[l * DPB_MAX_CHILDREN + j];
        __syncthreads();
        for (int j = threadIdx.x; j < nch; j += blockDim.x) {  // generators are distinct
            int rank = 0;
            for (int i = 0; i < nch; ++i) rank += gen[i] < gen[j];
            gsort[rank] = gen[j];
        }
        __syncthreads();
        // pair (b, j) -> child par[b] ^ gen[j]; it is a repeat when an earlier
        // parent b' < b reaches the same child, i.e. child ^ par[b'] is a generator
        const int n = np * nch;
        for (int i = warp; i < n; i += kSearchWarps) {
            const int b = i / nch;
            const uint32_t c = par[b] ^ gen[i - b * nch];
            bool rep = false;
            for (int bb = lane; bb < b; bb += 32) {
                const uint32_t v = c ^ par[bb];
                int lo = 0, hi = nch - 1;
                while (lo < hi) {
                    const int mid = (lo + hi) >> 1;
                    if (gsort[mid] < v) lo = mid + 1; else hi = mid;
                }
                rep |= gsort[lo] == v;
            }
            rep = __any_sync(kFull, rep);
            float s = 0.f;
            if (!rep) {
                for (int io = lane; io < d; io += 32) s += flip(xs[io], sign31(Ms[io], c));
                s = warp_sum(s) * a.inv_sqrt_d;
                if (c < (uint32_t)d) s = xs[c];  // basis override (Eq. 2); not reached by the level rule
            }
            if (lane == 0) {
                cid[i] = c;
                if (rep) {
                    zb[i] = -1.f;
                } else {
                    if ((int64_t)c < a.m) add_moments(a.acc, a.m, c, (double)s);
                    zb[i] = fabsf(z_of(s, c, a));
                }
            }
        }
        __syncthreads();
        if (l + 1 < a.levels)
            np = select_top(
                n, a.keep[l], zb, [&](int i) { return prio(zb[i], cid[i]); }, par, red, red + kSearchWarps,
                cid);
    }
}

// ---- the EMA step -----------------------------------------------------------------

__global__ void stats_update_kernel(double *acc, int64_t m, double alpha, float *mu, float *sigma) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += (int64_t)gridDim.x * blockDim.x) {
        const double n = acc[i];
        if (n < 0.5) continue;  // untouched: the sums are already zero
        const double s = acc[m + i], q = acc[2 * m + i];
        const double mean = s / n;
        const double mu0 = mu[i];
        mu[i] = (float)(mu0 + alpha * (mean - mu0));
        if (n >= 1.5) {
            const double var = q / n - mean * mean;
            const double v = sqrt(var > 0.0 ? var : 0.0);
            const double sg0 = sigma[i];
            sigma[i] = (float)(sg0 + alpha * (v - sg0));
        }
        acc[i] = 0.0;
        acc[m + i] = 0.0;
        acc[2 * m + i] = 0.0;
    }
}

int search_cap(const dpb_plan *p, const int *keep) {
    int cap = p->cfg.d;
    for (int l = 1; l < p->cfg.levels; ++l) {
        const int n = keep[l - 1] * p->cfg.children[l];
        if (n > cap) cap = n;
    }
    return cap;
}

size_t search_smem(int d, int cap) {
    return sizeof(uint32_t) * (2 * (size_t)d + kMaxKeep + 2 * DPB_MAX_CHILDREN + kSearchWarps + 4 + 2 * (size_t)cap);
}

void keep_of(const dpb_plan *p, int *keep) {
    for (int l = 0; l < DPB_MAX_LEVELS; ++l)
        keep[l] = p->cfg.select_mode == DPB_SELECT_PER_LEVEL ? p->cfg.k_per_level[l] : p->cfg.beam;
}

}  // namespace

bool stats_supported(const dpb_plan *p, size_t *smem_out) {
    int keep[DPB_MAX_LEVELS];
    keep_of(p, keep);
    for (int l = 0; l < p->cfg.levels; ++l)
        if (keep[l] < 1 || keep[l] > kMaxKeep) return false;
    const size_t smem = search_smem(p->cfg.d, search_cap(p, keep));
    if (smem_out) *smem_out = smem;
    return smem <= (size_t)kMaxSmemPerBlock;
}

cudaError_t launch_stats_accumulate(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                                    const float *sigma, const int32_t *sample, int32_t n_sample, double *acc,
                                    int32_t *status, cudaStream_t stream) {
    const int d = p->cfg.d;
    const int64_t m = (int64_t)p->m_mask + 1;
    if (T > 0) {
        const dim3 grid((unsigned)((T + kColRows - 1) / kColRows), (unsigned)((d + kColThreads - 1) / kColThreads));
        if (p->cfg.dtype == DPB_BF16)
            stats_columns_kernel<__nv_bfloat16><<<grid, kColThreads, 0, stream>>>(
                static_cast<const __nv_bfloat16 *>(x), T, d, acc, m);
        else
            stats_columns_kernel<float><<<grid, kColThreads, 0, stream>>>(static_cast<const float *>(x), T, d,
                                                                          acc, m);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (n_sample == 0 || p->cfg.levels < 2) return cudaSuccess;
    StatsArgs a{};
    a.x = x;
    a.T = T;
    a.d = d;
    a.levels = p->cfg.levels;
    keep_of(p, a.keep);
    for (int l = 0; l < DPB_MAX_LEVELS; ++l) a.children[l] = p->cfg.children[l];
    a.M = p->dM;
    a.G = p->dG;
    a.mu = mu;
    a.sigma = sigma;
    a.sample = sample;
    a.acc = acc;
    a.m = m;
    a.inv_sqrt_d = p->inv_sqrt_d;
    a.cap = search_cap(p, a.keep);
    a.status = status;
    const size_t smem = search_smem(d, a.cap);
    if (p->cfg.dtype == DPB_BF16) {
        cudaError_t e = cudaFuncSetAttribute(stats_search_kernel<__nv_bfloat16>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        stats_search_kernel<__nv_bfloat16><<<n_sample, kSearchThreads, smem, stream>>>(a);
    } else {
        cudaError_t e = cudaFuncSetAttribute(stats_search_kernel<float>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        stats_search_kernel<float><<<n_sample, kSearchThreads, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_stats_update(const dpb_plan *p, double *acc, float alpha, float *mu, float *sigma,
                                cudaStream_t stream) {
    const int64_t m = (int64_t)p->m_mask + 1;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, p->device);
    const int64_t want = (m + 255) / 256, cap = (int64_t)sms * 8;
    stats_update_kernel<<<(unsigned)(want < cap ? want : cap), 256, 0, stream>>>(acc, m, (double)alpha, mu, sigma);
    return cudaGetLastError();
}

}  // namespace dpb
