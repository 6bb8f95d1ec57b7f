// dpb_encode_mma.cu -- the §2.2 encoder with the child scoring of Eq. 6 on the
// tensor cores (bf16 inputs, beam 8, 16 children per parent).
//
// A warp owns two tokens at a time. At level l its 16 tensor-core rows are the
// (token, beam slot) pairs and the contraction is
//     score[row][j] = sum_iota (x_token (.) phi~_parent)[iota] * gamma_j[iota],
// i.e. rows x (.) phi~_p times the universal matrix Gamma_l (Eq. 6), with
// mma.sync m16n8k16 (bf16 x bf16 -> fp32). The A operand is never staged:
// each lane builds its fragment in registers as the bf16 bits of x XOR a sign
// mask. The K order is permuted so that the lane with q4 = lane % 4 holds the
// coordinates q4 + 4j of every 32-coordinate block, paired (j, j+4): the two
// sign bits of a pair sit 16 apart in the parent's sign word over the block,
// and one shift moves both to the bf16 sign positions 15 and 31. The sign
// word of parent p over block m is
//     W5[p & 31] ^ PQ[m][(p_lo >> 5) & 31] ^ XOR_k VH_k[m][chunk_k(p_hi)],
// the Walsh, block-parity and inverse-coordinate parts of parity(M[iota] & p)
// (App. A.4 Eq. 26). Gamma_l lives in shared memory in B-fragment order.
//
// Selection per token (global mode): level 0 keeps its exact top k, whose
// first 8 are the beam; level l keeps the first 8 of its distinct children
// (a tournament over the warp) and appends to a pool every child that is
// ahead of the pool's k-th entry; the code is the first k of the pool, sorted.
// Everything a child can displace is in the pool, so the code equals the top
// k over every candidate visited.
#include <algorithm>

#include "dpb_device.cuh"
#include "dpb_internal.h"
#include "dpb_select.cuh"

namespace dpb {

namespace {

constexpr int kWarps = 8;
constexpr int kBeam = 8;
constexpr int kPoolCap = 384;  // per token: k <= 256 plus one level's 128 children

struct EncMmaArgs {
    const __nv_bfloat16 *x;
    int64_t T;
    const float *mu, *sigma;
    int32_t *idx;
    float *val, *xnorm;
    int32_t *status;
    const uint32_t *frag, *G, *VH, *DD;
    int d, nblk, levels, k, t;
    float inv_sqrt_d;
};

// ---- shared-memory layout (32-bit words) ------------------------------------------

__host__ __device__ constexpr int block_words(int levels, int nblk, int nkc) {
    // frag [(L-1)][nblk][32][8], W5 [32], PQ [32][32], VH [nkc][32][32],
    // DD [(L-1)][kDedupSlots][2], G [L][16]
    return (levels - 1) * nblk * 256 + 32 + 1024 + nkc * 1024 + (levels - 1) * kDedupSlots * 2 + 8 * 16;
}

__host__ __device__ constexpr int warp_words(int nblk) {
    // x tile [2][nblk * 16], beams [2][8], pools z/id [2][kPoolCap] each,
    // duplicate bits [2][4], scratch [8], meta [8]
    return 2 * nblk * 16 + 16 + 4 * kPoolCap + 8 + 8 + 8;
}

struct WarpSmem {
    uint32_t *xt;
    uint32_t *beam;
    float *pz;
    uint32_t *pid;
    uint32_t *dup;
    float *scratch;
    int *meta;  // nbeam[2], npool[2], tau_key[2], tau_idx[2]
};

// ---- helpers ----------------------------------------------------------------------

__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Byte offsets of parent p into PQ[m] and VH_k[m], packed four to a word.
struct ParentOff {
    uint32_t w5;  // the Walsh word (the same for every block)
    uint32_t o;   // PQ, VH_0, VH_1, VH_2 byte offsets
    uint32_t o3;  // VH_3 byte offset
};

__device__ __forceinline__ ParentOff parent_offsets(uint32_t p, int t, const uint32_t *w5) {
    ParentOff po;
    po.w5 = w5[p & 31u];  // t >= 5: bits 0..4 belong to p_lo
    const uint32_t b1 = (((p & ((1u << t) - 1u)) >> 5) & 31u) * 4u;
    const uint32_t h0 = ((p >> t) & 31u) * 4u, h1 = ((p >> (t + 5)) & 31u) * 4u;
    const uint32_t h2 = ((p >> min(t + 10, 31)) & 31u) * 4u;
    const uint32_t h3 = ((p >> min(t + 15, 31)) & 31u) * 4u;
    po.o = b1 | (h0 << 8) | (h1 << 16) | (h2 << 24);
    po.o3 = h3;
    return po;
}

// Sign word of a parent over 32-coordinate block m (bit l = 1: coordinate
// 32 m + l of phi~_p is negative).
template <int NKC>
__device__ __forceinline__ uint32_t parent_signs(const ParentOff &po, const uint32_t *pq, const uint32_t *vh, int m) {
    const char *P = reinterpret_cast<const char *>(pq + m * 32);
    const char *V = reinterpret_cast<const char *>(vh + m * 32);
    uint32_t s = po.w5 ^ *reinterpret_cast<const uint32_t *>(P + __byte_perm(po.o, 0, 0x4440)) ^
                 *reinterpret_cast<const uint32_t *>(V + __byte_perm(po.o, 0, 0x4441));
    s ^= *reinterpret_cast<const uint32_t *>(V + 4096 + __byte_perm(po.o, 0, 0x4442));
    if (NKC > 2) s ^= *reinterpret_cast<const uint32_t *>(V + 8192 + __byte_perm(po.o, 0, 0x4443));
    if (NKC > 3) s ^= *reinterpret_cast<const uint32_t *>(V + 12288 + po.o3);
    return s;
}

// Coordinate i of one token's row, read back from the permuted tile.
__device__ __forceinline__ float x_at(const uint16_t *xh, int i) {
    const int m = i >> 5, l = i & 31;
    return __uint_as_float((uint32_t)xh[(m * 16 + (l & 3) * 4 + ((l >> 2) & 3)) * 2 + (l >> 4)] << 16);
}

// z = (s - mu_c) / sigma_c (§2.2 score standardisation); identity without tables.
__device__ __forceinline__ float standardise(float s, uint32_t c, const float *mu, const float *sigma,
                                             int32_t *status) {
    if (!mu) return s;
    const float sd = sigma[c];
    if (status && !(sd > 0.f)) set_status(status, DPB_DEV_BAD_SIGMA);
    return (s - mu[c]) / sd;
}

// Appends the lane-distributed entries with `take` set to a shared list at
// position n; returns the new length (warp-uniform).
__device__ __forceinline__ int warp_append(float *z, uint32_t *id, int n, bool take, float zv, uint32_t iv) {
    const int lane = threadIdx.x & 31;
    const unsigned mb = __ballot_sync(kFull, take);
    if (take) {
        const int pos = n + __popc(mb & ((1u << lane) - 1u));
        z[pos] = zv;
        id[pos] = iv;
    }
    return n + __popc(mb);
}

// Level 0 of one token: every coordinate is a candidate. Leaves the exact
// top k in the pool (unordered, n = k), its k-th entry in (tau_key, tau_idx),
// and the first 8 indices in `beam`.
__device__ __forceinline__ void level0(const EncMmaArgs &a, const uint16_t *xh, float *pz, uint32_t *pid,
                                       uint32_t *beam, float *scratch, uint32_t &tau_key, uint32_t &tau_idx) {
    const int lane = threadIdx.x & 31, d = a.d, k = a.k;
    const int lowbit = a.mu ? 0 : 16;  // keys of unstandardised bf16 values have 16 zero bits
    // Each lane's R-th best key: at least 32 R >= k candidates are at or above
    // the smallest of them, so that threshold loses nothing of the top k.
    const int R = (k + 31) >> 5;
    uint32_t best[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) best[r] = 0u;
    for (int i = lane; i < d; i += 32) {
        uint32_t kv = akey(standardise(x_at(xh, i), (uint32_t)i, a.mu, a.sigma, a.status)) + 1u;
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            if (r < R && kv > best[r]) {
                const uint32_t tmp = best[r];
                best[r] = kv;
                kv = tmp;
            }
        }
    }
    uint32_t mine = 0;
#pragma unroll
    for (int r = 0; r < 8; ++r)
        if (r == R - 1) mine = best[r];
    const uint32_t tau_low = __reduce_min_sync(kFull, mine);
    int n = 0;
    bool overflow = false;
    for (int i0 = 0; i0 < d && !overflow; i0 += 32) {
        const int i = i0 + lane;
        float z = 0.f;
        bool take = false;
        if (i < d) {
            z = standardise(x_at(xh, i), (uint32_t)i, a.mu, a.sigma, nullptr);
            take = akey(z) + 1u >= tau_low;
        }
        if (n + __popc(__ballot_sync(kFull, take)) > kPoolCap) {
            overflow = true;  // many equal keys at the threshold
        } else {
            n = warp_append(pz, pid, n, take, z, (uint32_t)i);
        }
    }
    __syncwarp();
    if (overflow) {
        // Exact k-th key over the whole row by bisection, then every entry
        // above it and the first ties by index.
        uint32_t tau = 0;
        for (int b = 30; b >= lowbit; --b) {
            const uint32_t c = tau | (1u << b);
            int cnt = 0;
            for (int i = lane; i < d; i += 32)
                cnt += akey(standardise(x_at(xh, i), (uint32_t)i, a.mu, a.sigma, nullptr)) >= c;
            if (__reduce_add_sync(kFull, cnt) >= k) tau = c;
        }
        n = 0;
        for (int i0 = 0; i0 < d; i0 += 32) {
            const int i = i0 + lane;
            float z = 0.f;
            if (i < d) z = standardise(x_at(xh, i), (uint32_t)i, a.mu, a.sigma, nullptr);
            n = warp_append(pz, pid, n, i < d && akey(z) > tau, z, (uint32_t)i);
        }
        for (int i0 = 0; i0 < d && n < k; i0 += 32) {
            const int i = i0 + lane;
            float z = 0.f;
            bool tie = false;
            if (i < d) {
                z = standardise(x_at(xh, i), (uint32_t)i, a.mu, a.sigma, nullptr);
                tie = akey(z) == tau;
            }
            const unsigned mb = __ballot_sync(kFull, tie);
            const int rank = __popc(mb & ((1u << lane) - 1u));
            if (tie && n + rank < k) {
                pz[n + rank] = z;
                pid[n + rank] = (uint32_t)i;
            }
            n = min(k, n + __popc(mb));
        }
        __syncwarp();
    }
    warp_kth(pz, pid, n, k, lowbit, tau_key, tau_idx);
    n = warp_compact_keep(pz, pid, n, tau_key, tau_idx);
    // the beam: the first 8 of the pool
    uint32_t bk, bi;
    warp_kth(pz, pid, n, kBeam, lowbit, bk, bi);
    int nb = 0;
    for (int e0 = 0; e0 < n; e0 += 32) {
        const int e = e0 + lane;
        const bool take = e < n && keeps(pz[e], pid[e], bk, bi);
        nb = warp_append(scratch, beam, nb, take, take ? pz[e] : 0.f, take ? pid[e] : 0u);
    }
    __syncwarp();
}

// Makes room in a token's pool for `incoming` entries: when they would not
// fit, the pool is cut to its first k (which raises its threshold).
__device__ __forceinline__ void pool_make_room(const WarpSmem &w, int tk, int k, int incoming) {
    const int n = w.meta[2 + tk];
    if (n + incoming <= kPoolCap) return;
    float *pz = w.pz + tk * kPoolCap;
    uint32_t *pid = w.pid + tk * kPoolCap;
    uint32_t tk_key, tk_idx;
    warp_kth(pz, pid, n, k, 0, tk_key, tk_idx);
    const int m = warp_compact_keep(pz, pid, n, tk_key, tk_idx);
    if ((threadIdx.x & 31) == 0) {
        w.meta[2 + tk] = m;
        w.meta[4 + tk] = (int)tk_key;
        w.meta[6 + tk] = (int)tk_idx;
    }
    __syncwarp();
}

// ---- the kernel ---------------------------------------------------------------------

template <int NKC>
__global__ void __launch_bounds__(kWarps * 32, 1) encode_mma_kernel(EncMmaArgs a) {
    extern __shared__ __align__(16) uint32_t smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int d = a.d, nblk = a.nblk, L = a.levels, k = a.k, t = a.t;
    const int q4 = lane & 3, slot = lane >> 2;

    uint32_t *s_frag = smem;
    uint32_t *s_w5 = s_frag + (L - 1) * nblk * 256;
    uint32_t *s_pq = s_w5 + 32;
    uint32_t *s_vh = s_pq + 1024;
    uint32_t *s_dd = s_vh + NKC * 1024;
    uint32_t *s_g = s_dd + (L - 1) * kDedupSlots * 2;
    {
        const uint4 *src = reinterpret_cast<const uint4 *>(a.frag);
        uint4 *dst = reinterpret_cast<uint4 *>(s_frag);
        for (int i = threadIdx.x; i < (L - 1) * nblk * 64; i += blockDim.x) dst[i] = src[i];
        for (int v = threadIdx.x; v < 32; v += blockDim.x) {
            uint32_t word = 0;
            for (int l = 0; l < 32; ++l) word |= (uint32_t)(__popc(l & v) & 1) << l;
            s_w5[v] = word;
        }
        for (int i = threadIdx.x; i < 1024; i += blockDim.x) s_pq[i] = (__popc((i >> 5) & i & 31) & 1) ? ~0u : 0u;
        for (int i = threadIdx.x; i < NKC * 1024; i += blockDim.x) s_vh[i] = a.VH[i];
        for (int i = threadIdx.x; i < (L - 1) * kDedupSlots * 2; i += blockDim.x) s_dd[i] = a.DD[i];
        for (int i = threadIdx.x; i < L * 16; i += blockDim.x) s_g[i] = a.G[(i >> 4) * DPB_MAX_CHILDREN + (i & 15)];
    }
    __syncthreads();

    WarpSmem w;
    {
        uint32_t *base = smem + block_words(L, nblk, NKC) + warp * warp_words(nblk);
        w.xt = base;
        w.beam = w.xt + 2 * nblk * 16;
        w.pz = reinterpret_cast<float *>(w.beam + 16);
        w.pid = reinterpret_cast<uint32_t *>(w.pz + 2 * kPoolCap);
        w.dup = w.pid + 2 * kPoolCap;
        w.scratch = reinterpret_cast<float *>(w.dup + 8);
        w.meta = reinterpret_cast<int *>(w.scratch + 8);
    }
    const int64_t npairs = (a.T + 1) / 2;

    for (int64_t pr = (int64_t)blockIdx.x * kWarps + warp; pr < npairs; pr += (int64_t)gridDim.x * kWarps) {
        const int64_t t0 = 2 * pr;
        const int ntok = t0 + 1 < a.T ? 2 : 1;

        // ---- both rows into the permuted tile; |x| ----
        uint16_t *xh = reinterpret_cast<uint16_t *>(w.xt);
        for (int tk = 0; tk < 2; ++tk) {
            const bool live = tk < ntok;
            const uint4 *row = reinterpret_cast<const uint4 *>(a.x + (t0 + (live ? tk : 0)) * d);
            float ss = 0.f;
            for (int ch = lane; ch < nblk * 4; ch += 32) {
                const uint4 v = live ? row[ch] : make_uint4(0u, 0u, 0u, 0u);
                const uint32_t words[4] = {v.x, v.y, v.z, v.w};
                const int m = ch >> 2, l0 = (ch & 3) * 8, half = l0 >> 4, pb = (l0 & 15) >> 2;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const uint16_t bits = (uint16_t)(words[e >> 1] >> (16 * (e & 1)));
                    xh[(tk * nblk * 16 + m * 16 + (e & 3) * 4 + pb + (e >> 2)) * 2 + half] = bits;
                    const float xf = __uint_as_float((uint32_t)bits << 16);
                    ss = fmaf(xf, xf, ss);
                }
            }
            ss = warp_sum(ss);
            if (live && lane == 0 && a.xnorm) a.xnorm[t0 + tk] = sqrtf(ss);
        }
        __syncwarp();

        // ---- level 0 ----
        for (int tk = 0; tk < ntok; ++tk) {
            uint32_t tau_key, tau_idx;
            level0(a, xh + tk * nblk * 32, w.pz + tk * kPoolCap, w.pid + tk * kPoolCap, w.beam + tk * 8,
                   w.scratch, tau_key, tau_idx);
            if (lane == 0) {
                w.meta[tk] = kBeam;
                w.meta[2 + tk] = k;
                w.meta[4 + tk] = (int)tau_key;
                w.meta[6 + tk] = (int)tau_idx;
            }
            __syncwarp();
        }
        if (ntok == 1 && lane == 0) w.meta[1] = 0;
        __syncwarp();

        // ---- levels 1 .. L-1 ----
        for (int l = 1; l < L; ++l) {
            const uint32_t *frag = s_frag + (l - 1) * nblk * 256;
            // this lane's tensor-core rows: (token 0, slot) and (token 1, slot)
            const uint32_t p0 = slot < w.meta[0] ? w.beam[slot] : 0u;
            const uint32_t p1 = slot < w.meta[1] ? w.beam[8 + slot] : 0u;
            const ParentOff o0 = parent_offsets(p0, t, s_w5), o1 = parent_offsets(p1, t, s_w5);
            float acc[2][2][4];
#pragma unroll
            for (int u = 0; u < 2; ++u)
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int r = 0; r < 4; ++r) acc[u][h][r] = 0.f;
            const uint4 *xa = reinterpret_cast<const uint4 *>(w.xt) + q4;
            const uint4 *xb = reinterpret_cast<const uint4 *>(w.xt + nblk * 16) + q4;
            const uint4 *fr = reinterpret_cast<const uint4 *>(frag) + lane * 2;
            const int sh = 15 - q4;
#pragma unroll 2
            for (int m = 0; m < nblk; ++m) {
                const uint4 va = xa[m * 4], vb = xb[m * 4];
                const uint32_t s0 = parent_signs<NKC>(o0, s_pq, s_vh, m);
                const uint32_t s1 = parent_signs<NKC>(o1, s_pq, s_vh, m);
                const uint4 f0 = fr[m * 64], f1 = fr[m * 64 + 1];
                // chunk 0 holds pairs 0 and 1 of the block, chunk 1 pairs 2 and 3
                const uint32_t a00 = va.x ^ ((s0 << sh) & 0x80008000u);
                const uint32_t a01 = vb.x ^ ((s1 << sh) & 0x80008000u);
                const uint32_t a02 = va.y ^ ((s0 << (sh - 4)) & 0x80008000u);
                const uint32_t a03 = vb.y ^ ((s1 << (sh - 4)) & 0x80008000u);
                const uint32_t a10 = va.z ^ ((s0 << (sh - 8)) & 0x80008000u);
                const uint32_t a11 = vb.z ^ ((s1 << (sh - 8)) & 0x80008000u);
                const uint32_t a12 = va.w ^ ((s0 << (sh - 12)) & 0x80008000u);
                const uint32_t a13 = vb.w ^ ((s1 << (sh - 12)) & 0x80008000u);
                float(&cc)[2][4] = acc[m & 1];
                mma_bf16(cc[0], a00, a01, a02, a03, f0.x, f0.y);
                mma_bf16(cc[1], a00, a01, a02, a03, f0.z, f0.w);
                mma_bf16(cc[0], a10, a11, a12, a13, f1.x, f1.y);
                mma_bf16(cc[1], a10, a11, a12, a13, f1.z, f1.w);
            }
            // accumulator (n-half h, register r): row slot (r < 2) or slot + 8
            // (r >= 2), child 8 h + 2 q4 + (r & 1)
            float sc[2][4];  // [token][2 h + (r & 1)]
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int r = 0; r < 4; ++r) sc[r >> 1][2 * h + (r & 1)] = (acc[0][h][r] + acc[1][h][r]) * a.inv_sqrt_d;
            const uint32_t *gl = s_g + l * 16;
            const uint32_t *ddl = s_dd + (l - 1) * kDedupSlots * 2;
            for (int tk = 0; tk < ntok; ++tk) {
                const int nb = w.meta[tk];
                const uint32_t *beam = w.beam + tk * 8;
                // ---- duplicate children (R8): p_s ^ g_j' == p_s' ^ g_j with s' < s
                // exactly when p_s ^ p_s' == g_j ^ g_j'; slot s's copy is dropped
                if (lane < 4) w.dup[tk * 4 + lane] = 0u;
                __syncwarp();
                if (lane < 28) {
                    int s = 1, sp = lane;  // the lane-th pair (sp, s), sp < s
                    while (sp >= s) {
                        sp -= s;
                        ++s;
                    }
                    if (s < nb) {
                        const uint32_t delta = beam[s] ^ beam[sp];
                        uint32_t h = dedup_hash(delta);
                        for (int probe = 0; probe < kDedupSlots; ++probe) {
                            const uint32_t key = ddl[2 * h];
                            if (key == 0u) break;
                            if (key == delta + 1u) {
                                const uint32_t bit = (uint32_t)s * 16u + (ddl[2 * h + 1] & 0xffu);
                                atomicOr(&w.dup[tk * 4 + (bit >> 5)], 1u << (bit & 31u));
                            }
                            h = (h + 1u) & (kDedupSlots - 1);
                        }
                    }
                }
                __syncwarp();
                // ---- this lane's 4 children of token tk
                const uint32_t p = tk == 0 ? p0 : p1;
                const bool live = slot < nb;
                Cand c[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = 8 * (e >> 1) + 2 * q4 + (e & 1);
                    const uint32_t ci = p ^ gl[j];
                    const uint32_t bit = (uint32_t)slot * 16u + (uint32_t)j;
                    const bool dup = (w.dup[tk * 4 + (bit >> 5)] >> (bit & 31u)) & 1u;
                    const float z = standardise(tk == 0 ? sc[0][e] : sc[1][e], ci, a.mu, a.sigma, live ? a.status : nullptr);
                    c[e].idx = ci;
                    c[e].z = z;
                    c[e].key = (live && !dup) ? akey(z) + 1u : 0u;
                }
                // ---- pool: every child ahead of the pool's k-th entry
                float *pz = w.pz + tk * kPoolCap;
                uint32_t *pid = w.pid + tk * kPoolCap;
                {
                    const uint32_t tkey = (uint32_t)w.meta[4 + tk], tidx = (uint32_t)w.meta[6 + tk];
                    int cnt = 0;
#pragma unroll
                    for (int e = 0; e < 4; ++e) cnt += c[e].key != 0u && keeps(c[e].z, c[e].idx, tkey, tidx);
                    pool_make_room(w, tk, k, __reduce_add_sync(kFull, cnt));
                }
                {
                    const uint32_t tkey = (uint32_t)w.meta[4 + tk], tidx = (uint32_t)w.meta[6 + tk];
                    int n = w.meta[2 + tk];
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        n = warp_append(pz, pid, n, c[e].key != 0u && keeps(c[e].z, c[e].idx, tkey, tidx), c[e].z,
                                        c[e].idx);
                    __syncwarp();
                    if (lane == 0) w.meta[2 + tk] = n;
                }
                // ---- the beam of level l
                if (l + 1 < L) {
                    const int nbn = warp_tournament4(c, kBeam, w.scratch, w.beam + tk * 8);
                    if (lane == 0) w.meta[tk] = nbn;
                }
                __syncwarp();
            }
        }

        // ---- the code of each token: the first k of its pool, sorted ----
        int cap = 32;
        while (cap < k) cap <<= 1;
        for (int tk = 0; tk < ntok; ++tk) {
            float *pz = w.pz + tk * kPoolCap;
            uint32_t *pid = w.pid + tk * kPoolCap;
            int n = w.meta[2 + tk];
            uint32_t kk, ki;
            warp_kth(pz, pid, n, k, 0, kk, ki);
            n = warp_compact_keep(pz, pid, n, kk, ki);
            warp_sort(pz, pid, n, cap);
            const int64_t row = t0 + tk;
            for (int e = lane; e < k; e += 32) {
                a.idx[row * k + e] = (int32_t)pid[e];
                a.val[row * k + e] = pz[e];
            }
            __syncwarp();
        }
    }
}

template <int NKC>
cudaError_t run(const dpb_plan *p, const EncMmaArgs &a, cudaStream_t stream) {
    const size_t smem = encode_mma_smem(p);
    const cudaError_t e =
        cudaFuncSetAttribute(encode_mma_kernel<NKC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, p->device);
    const int64_t pairs = (a.T + 1) / 2;
    const int grid = (int)std::min<int64_t>((pairs + kWarps - 1) / kWarps, (int64_t)std::max(sms, 1));
    encode_mma_kernel<NKC><<<grid, kWarps * 32, smem, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace

size_t encode_mma_smem(const dpb_plan *p) {
    const int nblk = p->cfg.d / 32, nkc = std::max(2, p->kvh);
    return sizeof(uint32_t) * ((size_t)block_words(p->cfg.levels, nblk, nkc) + (size_t)kWarps * warp_words(nblk));
}

cudaError_t launch_encode_mma(const dpb_plan *p, const void *x, int64_t T, const float *mu,
                              const float *sigma, int32_t *idx, float *val, float *xnorm,
                              int32_t *status, cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    EncMmaArgs a{};
    a.x = static_cast<const __nv_bfloat16 *>(x);
    a.T = T;
    a.mu = mu;
    a.sigma = sigma;
    a.idx = idx;
    a.val = val;
    a.xnorm = xnorm;
    a.status = status;
    a.frag = p->dFRAG;
    a.G = p->dG;
    a.VH = p->dVH;
    a.DD = p->dDD;
    a.d = c.d;
    a.nblk = c.d / 32;
    a.levels = c.levels;
    a.k = c.k;
    a.t = p->t;
    a.inv_sqrt_d = p->inv_sqrt_d;
    const int nkc = std::max(2, p->kvh);
    if (nkc == 2) return run<2>(p, a, stream);
    if (nkc == 3) return run<3>(p, a, stream);
    return run<4>(p, a, stream);
}

}  // namespace dpb
