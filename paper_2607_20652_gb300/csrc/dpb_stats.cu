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
//              child's raw score to the sums. A thread scores one child:
//              per 32-coordinate block, the child's sign word (from the
//              plan's per-block tables) indexes eight 16-entry tables of the
//              row's signed nibble sums (d <= 2048; a warp of popcounts per
//              child beyond).
//   update     a pass over the 2^N count words; only touched features read
//              their sums, move their moments and clear the sums.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "dpb_device.cuh"
#include "dpb_internal.h"
#include "dpb_lut.cuh"

namespace dpb {
namespace {

constexpr int kColThreads = 256;
constexpr int kColRows = 256;     // rows per block of the column pass
constexpr int kColChunk = 32;     // rows per fp32 partial before it joins the fp64 sums
constexpr int kSearchThreads = 512;
constexpr int kSearchWarps = kSearchThreads / 32;
constexpr int kMaxKeep = 64;
constexpr int kGenSlots = 512;    // open-addressing slots of one level's generator set
constexpr int kNibStride = 17;    // a nibble table: 16 sums + 1 pad word (bank spread)

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
    const uint32_t *VH2;  // [nkc][nblk][32] inverse-coordinate sign words (d <= 2048)
    int t;                // field degree
};

// Shared-memory carve-up of the search block (32-bit words).
struct SearchLayout {
    int xs, ms, th, vh, w5, par, gen, gslot, red, hist, zb, cid, words;
};

__host__ __device__ inline SearchLayout search_layout(int d, int nkc, int cap) {
    const int nblk = (d + 31) / 32;
    SearchLayout L{};
    int o = 0;
    L.xs = o, o += pad4(d);
    L.ms = o, o += nkc ? 0 : pad4(d);                        // M rows (popcount scoring)
    L.th = o, o += nkc ? pad4(nblk * 8 * kNibStride) : 0;    // nibble sums of the row
    L.vh = o, o += nkc * nblk * 32;
    L.w5 = o, o += 32;
    L.par = o, o += kMaxKeep;
    L.gen = o, o += DPB_MAX_CHILDREN;
    L.gslot = o, o += kGenSlots;
    L.red = o, o += 32;
    L.hist = o, o += 256;
    L.zb = o, o += cap;
    L.cid = o, o += cap;
    L.words = o;
    return L;
}

__device__ __forceinline__ uint32_t gen_hash(uint32_t v) { return (v * 2654435761u) >> 23; }  // 9 bits

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
// slot i's priority. The threshold is the keep-th largest priority, found one
// byte at a time from the top by 256-bin histograms (priorities are
// distinct, so exactly keep slots reach it).
template <typename PR>
__device__ int select_top(int n, int keep, const float *zb, PR pr, uint32_t *par, int *red, int *hist,
                          const uint32_t *cid) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int valid = 0;
    for (int i = tid; i < n; i += blockDim.x) valid += zb[i] >= 0.f;
    valid = block_sum(valid, red);
    const int K = keep < valid ? keep : valid;
    uint64_t tau = 0;
    if (K < valid) {
        int need = K;
        for (int shift = 56; shift >= 0; shift -= 8) {
            const uint64_t hi = shift == 56 ? 0ull : ~0ull << (shift + 8);
            for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0;
            __syncthreads();
            for (int i = tid; i < n; i += blockDim.x) {
                if (zb[i] < 0.f) continue;
                const uint64_t P = pr(i);
                if ((P & hi) == (tau & hi)) atomicAdd(&hist[(P >> shift) & 255u], 1);
            }
            __syncthreads();
            if (warp == 0) {
                // lane owns bins 255 - 8 lane - r, r < 8 (descending); counts above it
                int cnt[8], tot = 0;
#pragma unroll
                for (int r = 0; r < 8; ++r) tot += (cnt[r] = hist[255 - 8 * lane - r]);
                int incl = tot;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int v = __shfl_up_sync(kFull, incl, o);
                    if (lane >= o) incl += v;
                }
                int run = incl - tot;
                if (run < need && need <= incl) {
#pragma unroll
                    for (int r = 0; r < 8; ++r) {
                        if (run + cnt[r] >= need) {
                            red[kSearchWarps] = 255 - 8 * lane - r;
                            red[kSearchWarps + 1] = run;
                            break;
                        }
                        run += cnt[r];
                    }
                }
            }
            __syncthreads();
            tau |= (uint64_t)red[kSearchWarps] << shift;
            need -= red[kSearchWarps + 1];
            __syncthreads();
        }
    }
    int *cnt = red + kSearchWarps + 2;
    if (tid == 0) *cnt = 0;
    __syncthreads();
    for (int i = tid; i < n; i += blockDim.x)
        if (zb[i] >= 0.f && pr(i) >= tau) par[atomicAdd(cnt, 1)] = cid[i];
    __syncthreads();
    return K;
}

// NKC > 0: table-driven scoring (d <= 2048, NKC chunk tables); NKC == 0: a
// warp of popcounts per child.
template <typename Tio, int NKC>
__global__ void __launch_bounds__(kSearchThreads, 1) stats_search_kernel(StatsArgs a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int d = a.d, nblk = (d + 31) / 32;
    const SearchLayout L = search_layout(d, NKC, a.cap);
    float *xs = reinterpret_cast<float *>(smem + L.xs);
    uint32_t *Ms = smem + L.ms;
    float *TH = reinterpret_cast<float *>(smem + L.th);
    uint32_t *vh = smem + L.vh;
    uint32_t *w5 = smem + L.w5;
    uint32_t *par = smem + L.par;
    uint32_t *gen = smem + L.gen;
    uint32_t *gslot = smem + L.gslot;
    int *red = reinterpret_cast<int *>(smem + L.red);
    int *hist = reinterpret_cast<int *>(smem + L.hist);
    float *zb = reinterpret_cast<float *>(smem + L.zb);  // |z| (-1: not a candidate)
    uint32_t *cid = smem + L.cid;                         // candidate index

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int32_t row = a.sample[blockIdx.x];
    if (row < 0 || row >= a.T) {
        if (tid == 0) set_status(a.status, DPB_DEV_BAD_INDEX);
        return;
    }
    const Tio *xr = static_cast<const Tio *>(a.x) + (int64_t)row * d;
    for (int i = tid; i < d; i += blockDim.x) {
        xs[i] = ld_elem(xr, i);
        if (NKC == 0) Ms[i] = a.M[i];
    }
    if (NKC > 0) {
        for (int i = tid; i < NKC * nblk * 32; i += blockDim.x) vh[i] = a.VH2[i];
        if (tid < 32) {
            uint32_t word = 0;
            for (int l = 0; l < 32; ++l) word |= (uint32_t)(__popc(l & tid) & 1) << l;
            w5[tid] = word;
        }
    }
    __syncthreads();
    if (NKC > 0) {
        // nibble table tau (coordinates 4 tau .. 4 tau + 3): entry v = sum_j (-1)^{v_j} x[4 tau + j]
        for (int tau = tid; tau < nblk * 8; tau += blockDim.x) {
            const int i0 = 4 * tau;
            const float h0 = i0 < d ? xs[i0] : 0.f, h1 = i0 + 1 < d ? xs[i0 + 1] : 0.f;
            const float h2 = i0 + 2 < d ? xs[i0 + 2] : 0.f, h3 = i0 + 3 < d ? xs[i0 + 3] : 0.f;
            const float A[4] = {h0 + h1, h1 - h0, h0 - h1, -h0 - h1};
            const float B[4] = {h2 + h3, h3 - h2, h2 - h3, -h2 - h3};
            float *T = TH + tau * kNibStride;
#pragma unroll
            for (int v = 0; v < 16; ++v) T[v] = A[v & 3] + B[v >> 2];
        }
    }
    // level 0: the basis coordinates
    for (int i = tid; i < d; i += blockDim.x) {
        zb[i] = fabsf(z_of(xs[i], (uint32_t)i, a));
        cid[i] = (uint32_t)i;
    }
    __syncthreads();
    auto pri = [&](int i) { return prio(zb[i], cid[i]); };
    int np = select_top(d, a.keep[0], zb, pri, par, red, hist, cid);

    for (int l = 1; l < a.levels; ++l) {
        const int nch = a.children[l];
        for (int j = tid; j < nch; j += blockDim.x) gen[j] = a.G[l * DPB_MAX_CHILDREN + j];
        for (int j = tid; j < kGenSlots; j += blockDim.x) gslot[j] = 0u;
        __syncthreads();
        // the level's generator set (distinct values; key g + 1, 0 = empty)
        for (int j = tid; j < nch; j += blockDim.x) {
            uint32_t h = gen_hash(gen[j]);
            for (int probe = 0; probe < kGenSlots; ++probe) {
                if (atomicCAS(&gslot[h], 0u, gen[j] + 1u) == 0u) break;
                h = (h + 1u) & (kGenSlots - 1);
            }
        }
        __syncthreads();
        // pair (b, j) -> child par[b] ^ gen[j]; a repeat when an earlier parent
        // b' < b reaches the same child, i.e. child ^ par[b'] is a generator
        auto repeat = [&](uint32_t c, int b) {
            for (int bb = 0; bb < b; ++bb) {
                const uint32_t v = c ^ par[bb];
                uint32_t h = gen_hash(v);
                for (int probe = 0; probe < kGenSlots; ++probe) {
                    const uint32_t e = gslot[h];
                    if (e == 0u) break;
                    if (e == v + 1u) return true;
                    h = (h + 1u) & (kGenSlots - 1);
                }
            }
            return false;
        };
        const int n = np * nch;
        if (NKC > 0) {
            for (int i = tid; i < n; i += blockDim.x) {
                const int b = i / nch;
                const uint32_t c = par[b] ^ gen[i - b * nch];
                cid[i] = c;
                if (repeat(c, b)) {
                    zb[i] = -1.f;
                    continue;
                }
                uint32_t o1, o2;
                code_offsets(c, a.t, w5, o1, o2);
                float acc = 0.f;
                for (int q = 0; q < nblk; ++q) {
                    const uint32_t sw = block_signs<(NKC > 1 ? NKC : 2)>(vh, nblk, q, o1, o2);
                    const float *T = TH + q * 8 * kNibStride;
                    float part = 0.f;
#pragma unroll
                    for (int k = 0; k < 8; ++k) part += T[k * kNibStride + ((sw >> (4 * k)) & 15u)];
                    acc += part;
                }
                float s = acc * a.inv_sqrt_d;
                if (c < (uint32_t)d) s = xs[c];  // basis override (Eq. 2); not reached by the level rule
                if ((int64_t)c < a.m) add_moments(a.acc, a.m, c, (double)s);
                zb[i] = fabsf(z_of(s, c, a));
            }
        } else {
            for (int i = warp; i < n; i += kSearchWarps) {
                const int b = i / nch;
                const uint32_t c = par[b] ^ gen[i - b * nch];
                const bool rep = lane == 0 && repeat(c, b);
                if (__shfl_sync(kFull, rep, 0)) {
                    if (lane == 0) {
                        cid[i] = c;
                        zb[i] = -1.f;
                    }
                    continue;
                }
                float s = 0.f;
                for (int io = lane; io < d; io += 32) s += flip(xs[io], sign31(Ms[io], c));
                s = warp_sum(s) * a.inv_sqrt_d;
                if (c < (uint32_t)d) s = xs[c];
                if (lane == 0) {
                    cid[i] = c;
                    if ((int64_t)c < a.m) add_moments(a.acc, a.m, c, (double)s);
                    zb[i] = fabsf(z_of(s, c, a));
                }
            }
        }
        __syncthreads();
        if (l + 1 < a.levels) np = select_top(n, a.keep[l], zb, pri, par, red, hist, cid);
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

template <typename Tio, int NKC>
cudaError_t run_search(const StatsArgs &a, int32_t n_sample, size_t smem, cudaStream_t stream) {
    const cudaError_t e = allow_smem((const void *)stats_search_kernel<Tio, NKC>, smem);
    if (e != cudaSuccess) return e;
    stats_search_kernel<Tio, NKC><<<n_sample, kSearchThreads, smem, stream>>>(a);
    return cudaGetLastError();
}

int search_cap(const dpb_plan *p, const int *keep) {
    int cap = p->cfg.d;
    for (int l = 1; l < p->cfg.levels; ++l) {
        const int n = keep[l - 1] * p->cfg.children[l];
        if (n > cap) cap = n;
    }
    return cap;
}

int search_nkc(const dpb_plan *p) { return p->cfg.d <= 2048 ? std::max(2, p->kvh) : 0; }

size_t search_smem(const dpb_plan *p, int cap) {
    return sizeof(uint32_t) * (size_t)search_layout(p->cfg.d, search_nkc(p), cap).words;
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
    const size_t smem = search_smem(p, search_cap(p, keep));
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
    a.VH2 = p->dVH2;
    a.t = p->t;
    const size_t smem = search_smem(p, a.cap);
    const int nkc = search_nkc(p);
    if (p->cfg.dtype == DPB_BF16) {
        if (nkc == 0) return run_search<__nv_bfloat16, 0>(a, n_sample, smem, stream);
        if (nkc == 2) return run_search<__nv_bfloat16, 2>(a, n_sample, smem, stream);
        if (nkc == 3) return run_search<__nv_bfloat16, 3>(a, n_sample, smem, stream);
        return run_search<__nv_bfloat16, 4>(a, n_sample, smem, stream);
    }
    if (nkc == 0) return run_search<float, 0>(a, n_sample, smem, stream);
    if (nkc == 2) return run_search<float, 2>(a, n_sample, smem, stream);
    if (nkc == 3) return run_search<float, 3>(a, n_sample, smem, stream);
    return run_search<float, 4>(a, n_sample, smem, stream);
}

cudaError_t launch_stats_update(const dpb_plan *p, double *acc, float alpha, float *mu, float *sigma,
                                cudaStream_t stream) {
    // one feature per thread: the touched features' dependent loads and fp64
    // arithmetic then all run at once instead of in a grid-stride chain
    const int64_t m = (int64_t)p->m_mask + 1;
    const int64_t blocks = (m + 255) / 256;
    stats_update_kernel<<<(unsigned)(blocks < 0x7fffffff ? blocks : 0x7fffffff), 256, 0, stream>>>(
        acc, m, (double)alpha, mu, sigma);
    return cudaGetLastError();
}

}  // namespace dpb
