// dpb_encode.cu -- the §2.2 encoder, one warp per token.
//
// Per token: level 0 takes the d coordinates as candidates (a coordinate read,
// Eq. 2); level l >= 1 takes the distinct children p ^ g_j of the previous
// beam and scores them through Eq. 6, <gamma_j, phi~_p (.) x>, with every sign
// generated on chip from parity(M[iota] AND .) (Eq. 26). The beam is the top
// B of a level; the code is the top k of every candidate, kept as a running
// top-k so a warp never holds more than k + B * Delta candidates.
#include <algorithm>

#include "dpb_device.cuh"
#include "dpb_internal.h"

namespace dpb {

namespace {

struct EncodeArgs {
    const void *x;
    int64_t T;
    const float *mu, *sigma;
    int32_t *idx;
    float *val, *xnorm;
    int32_t *status;
    const uint32_t *M, *G;
    int d, levels, beam, k, kmax0, list_cap, pool_cap, sort_cap;
    int children[DPB_MAX_LEVELS];
    float inv_sqrt_d;
};

// (mu_c, 1 / sigma_c) for every feature, read by the encoders in one 8-byte load.
__global__ void pack_tables_kernel(const float *mu, const float *sigma, float2 *tab, int64_t m) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += (int64_t)gridDim.x * blockDim.x)
        tab[i] = make_float2(mu[i], __frcp_rn(sigma[i]));
}

// z = (s - mu_c) / sigma_c (this general encoder scores in its own order, so
// its last bits need not match the tensor-core encoders' in any case)
__device__ __forceinline__ float standardise(float s, uint32_t c, const EncodeArgs &a, int32_t *status) {
    if (!a.mu) return s;
    const float sd = a.sigma[c];
    if (!(sd > 0.f)) set_status(status, DPB_DEV_BAD_SIGMA);
    return (s - a.mu[c]) / sd;
}

// Per-warp shared-memory carve-up (floats and words are both 4 bytes).
struct WarpSmem {
    float *xs, *xp;        // x row, x (.) phi~_p
    float *lz;             // level candidates (scores)
    uint32_t *lid;         // level candidates (indices)
    float *pz;             // pool: running top-k followed by a level
    uint32_t *pid;
    float *sz;             // selection output / sort buffer
    uint32_t *sid;
    uint32_t *beam;
};

template <typename Tin>
__global__ void __launch_bounds__(128) encode_warp_kernel(EncodeArgs a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int d = a.d;
    uint32_t *sM = smem;
    uint32_t *sG = sM + d;  // levels * 256 words
    for (int i = threadIdx.x; i < d; i += blockDim.x) sM[i] = a.M[i];
    for (int i = threadIdx.x; i < a.levels * DPB_MAX_CHILDREN; i += blockDim.x) sG[i] = a.G[i];
    __syncthreads();

    const size_t per_warp = 2 * (size_t)d + 2 * (size_t)a.list_cap + 2 * (size_t)a.pool_cap +
                            2 * (size_t)a.sort_cap + 32;
    uint32_t *base = sG + a.levels * DPB_MAX_CHILDREN + warp * per_warp;
    WarpSmem w;
    w.xs = reinterpret_cast<float *>(base);
    w.xp = w.xs + d;
    w.lz = w.xp + d;
    w.lid = reinterpret_cast<uint32_t *>(w.lz + a.list_cap);
    w.pz = reinterpret_cast<float *>(w.lid + a.list_cap);
    w.pid = reinterpret_cast<uint32_t *>(w.pz + a.pool_cap);
    w.sz = reinterpret_cast<float *>(w.pid + a.pool_cap);
    w.sid = reinterpret_cast<uint32_t *>(w.sz + a.sort_cap);
    w.beam = w.sid + a.sort_cap;

    const Tin *X = static_cast<const Tin *>(a.x);
    for (int64_t t = (int64_t)blockIdx.x * nwarps + warp; t < a.T; t += (int64_t)gridDim.x * nwarps) {
        // ---- load the row and its norm ----
        float ss = 0.f;
        for (int i = lane; i < d; i += 32) {
            const float v = ld_elem(X, t * d + i);
            w.xs[i] = v;
            ss += v * v;
        }
        ss = warp_sum(ss);
        if (a.xnorm && lane == 0) a.xnorm[t] = sqrtf(ss);

        // ---- level 0: every coordinate is a candidate ----
        for (int i = lane; i < d; i += 32) {
            w.lz[i] = standardise(w.xs[i], (uint32_t)i, a, a.status);
            w.lid[i] = (uint32_t)i;
        }
        __syncwarp();
        // the best max(B, k) of level 0, sorted: the beam is its head, the
        // running code its first k entries
        const int n0 = warp_select(w.lz, w.lid, d, a.kmax0, w.sz, w.sid);
        warp_sort(w.sz, w.sid, n0, a.sort_cap);
        int nbeam = min(a.beam, n0);
        for (int e = lane; e < nbeam; e += 32) w.beam[e] = w.sid[e];
        int nrun = min(a.k, n0);
        for (int e = lane; e < nrun; e += 32) {
            w.pz[e] = w.sz[e];
            w.pid[e] = w.sid[e];
        }
        __syncwarp();

        for (int l = 1; l < a.levels; ++l) {
            const int nch = a.children[l];
            const uint32_t *gl = sG + l * DPB_MAX_CHILDREN;
            // ---- score every (parent, generator) slot through Eq. 6 ----
            for (int b = 0; b < nbeam; ++b) {
                const uint32_t p = w.beam[b];
                for (int i = lane; i < d; i += 32) w.xp[i] = flip(w.xs[i], sign31(sM[i], p));
                __syncwarp();
                for (int j = 0; j < nch; ++j) {
                    const uint32_t g = gl[j];
                    float acc = 0.f;
                    for (int i = lane; i < d; i += 32) acc += flip(w.xp[i], sign31(sM[i], g));
                    acc = warp_sum(acc);
                    if (lane == 0) {
                        w.lz[b * nch + j] = acc * a.inv_sqrt_d;
                        w.lid[b * nch + j] = p ^ g;
                    }
                }
                __syncwarp();
            }
            // ---- keep each index once (the candidates form a set) ----
            const int nslot = nbeam * nch;
            int nu = 0;
            for (int s0 = 0; s0 < nslot; s0 += 32) {
                const int s = s0 + lane;
                bool keep = false;
                float z = 0.f;
                uint32_t c = 0;
                if (s < nslot) {
                    c = w.lid[s];
                    keep = true;
                    for (int r = 0; r < s; ++r)
                        if (w.lid[r] == c) keep = false;
                    z = standardise(w.lz[s], c, a, a.status);
                }
                const unsigned m = __ballot_sync(kFull, keep);
                if (keep) {
                    const int pos = nrun + nu + __popc(m & ((1u << lane) - 1u));
                    w.pz[pos] = z;
                    w.pid[pos] = c;
                }
                nu += __popc(m);
            }
            __syncwarp();
            // ---- beam of this level ----
            if (l + 1 < a.levels) {
                nbeam = warp_select(w.pz + nrun, w.pid + nrun, nu, a.beam, w.sz, w.sid);
                for (int e = lane; e < nbeam; e += 32) w.beam[e] = w.sid[e];
                __syncwarp();
            }
            // ---- running top-k over everything seen ----
            nrun = warp_select(w.pz, w.pid, nrun + nu, a.k, w.sz, w.sid);
            for (int e = lane; e < nrun; e += 32) {
                w.pz[e] = w.sz[e];
                w.pid[e] = w.sid[e];
            }
            __syncwarp();
        }

        // ---- the code, sorted ----
        for (int e = lane; e < nrun; e += 32) {
            w.sz[e] = w.pz[e];
            w.sid[e] = w.pid[e];
        }
        __syncwarp();
        warp_sort(w.sz, w.sid, nrun, a.sort_cap);
        if (nrun < a.k && lane == 0) set_status(a.status, DPB_DEV_SHORT_CODE);
        for (int e = lane; e < a.k; e += 32) {
            const bool ok = e < nrun;
            a.idx[t * a.k + e] = ok ? (int32_t)w.sid[e] : 0;
            a.val[t * a.k + e] = ok ? w.sz[e] : 0.f;
        }
        __syncwarp();
    }
}

int pow2_at_least(int v) {
    int p = 1;
    while (p < v) p <<= 1;
    return p;
}

void shape(const dpb_plan *p, int &list_cap, int &pool_cap, int &sort_cap, int &kmax0) {
    const dpb_config &c = p->cfg;
    int maxlvl = 0;
    for (int l = 1; l < c.levels; ++l) maxlvl = std::max(maxlvl, c.beam * c.children[l]);
    list_cap = std::max(c.d, maxlvl);   // level 0 lists d coordinates
    pool_cap = c.k + maxlvl;            // running top-k plus one level
    kmax0 = std::min(c.d, std::max(c.beam, c.k));
    // selection outputs (level-0 head, a beam, the running top-k) and the sorts
    sort_cap = std::max(32, pow2_at_least(std::max(kmax0, std::max(c.k, c.beam))));
}

}  // namespace

size_t encode_smem_header(const dpb_plan *p) {
    return sizeof(uint32_t) * ((size_t)p->cfg.d + (size_t)p->cfg.levels * DPB_MAX_CHILDREN);
}

size_t encode_smem_per_warp(const dpb_plan *p) {
    int list_cap, pool_cap, sort_cap, kmax0;
    shape(p, list_cap, pool_cap, sort_cap, kmax0);
    return sizeof(uint32_t) *
           (2 * (size_t)p->cfg.d + 2 * (size_t)list_cap + 2 * (size_t)pool_cap + 2 * (size_t)sort_cap + 32);
}

cudaError_t launch_encode(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                          const float *sigma, int32_t *idx, float *val, float *xnorm,
                          int32_t *status, float2 *tab_scratch, cudaStream_t stream) {
    // standardisation tables as (mu, 1 / sigma) pairs: one load per candidate
    const float2 *tab = nullptr;
    if (mu && tab_scratch) {
        const int64_t m = (int64_t)p->m_mask + 1;
        const int64_t want = (m + 255) / 256, cap = (int64_t)std::max(p->sms, 1) * 8;
        pack_tables_kernel<<<(unsigned)(want < cap ? want : cap), 256, 0, stream>>>(mu, sigma, tab_scratch, m);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        tab = tab_scratch;
    }
    // the paper's per-level selection: tcgen05 scoring
    if (p->cfg.select_mode == DPB_SELECT_PER_LEVEL)
        return launch_encode_pl(p, x, T, mu, sigma, tab, idx, val, xnorm, status, stream);
    // bf16 rows on 16-byte boundaries, beam <= 16, 16 children: tensor-core scoring
    if (p->mma_encode && (reinterpret_cast<uintptr_t>(x) & 15u) == 0)
        return launch_encode_mma(p, x, T, mu, sigma, tab, idx, val, xnorm, status, stream);
    const dpb_config &c = p->cfg;
    EncodeArgs a{};
    a.x = x;
    a.T = T;
    a.mu = mu;
    a.sigma = sigma;
    a.idx = idx;
    a.val = val;
    a.xnorm = xnorm;
    a.status = status;
    a.M = p->dM;
    a.G = p->dG;
    a.d = c.d;
    a.levels = c.levels;
    a.beam = c.beam;
    a.k = c.k;
    shape(p, a.list_cap, a.pool_cap, a.sort_cap, a.kmax0);
    for (int l = 0; l < DPB_MAX_LEVELS; ++l) a.children[l] = c.children[l];
    a.inv_sqrt_d = p->inv_sqrt_d;

    const size_t head = encode_smem_header(p), per_warp = encode_smem_per_warp(p);
    int warps = 4;
    while (warps > 1 && head + warps * per_warp > 200 * 1024) --warps;
    const size_t smem = head + warps * per_warp;
    const int64_t want = (T + warps - 1) / warps;
    const int grid = (int)std::min<int64_t>(want, (int64_t)std::max(p->sms, 1) * 16);
    if (c.dtype == DPB_BF16) {
        const cudaError_t e = allow_smem((const void *)encode_warp_kernel<__nv_bfloat16>, smem);
        if (e != cudaSuccess) return e;
        encode_warp_kernel<__nv_bfloat16><<<grid, warps * 32, smem, stream>>>(a);
    } else {
        const cudaError_t e = allow_smem((const void *)encode_warp_kernel<float>, smem);
        if (e != cudaSuccess) return e;
        encode_warp_kernel<float><<<grid, warps * 32, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace dpb
