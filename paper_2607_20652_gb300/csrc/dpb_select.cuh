// dpb_select.cuh -- warp-level exact selection for the encoder: the K first
// candidates in the order (|z| descending, index ascending) of §2.2's AbsTopK.
// Keys are the bit patterns of |z| (for finite floats they order like the
// values); a candidate list lives in shared memory as (z, index) pairs.
#pragma once

#include <cstdint>

#include "dpb_device.cuh"

namespace dpb {

// The K-th candidate (tau_key, tau_idx) of a list of n >= K entries. A
// candidate is among the first K iff key > tau_key, or key == tau_key and
// index <= tau_idx. `lowbit` is the lowest key bit that can be set (16 when
// the keys come from bf16 values). Bisection on the key bits, then on the
// index bits among ties, with counts reduced across the warp.
__device__ __forceinline__ void warp_kth(const float *z, const uint32_t *id, int n, int K, int lowbit,
                                         uint32_t &tau_key, uint32_t &tau_idx) {
    const int lane = threadIdx.x & 31;
    uint32_t tau = 0;
    for (int b = 30; b >= lowbit; --b) {
        const uint32_t c = tau | (1u << b);
        int cnt = 0;
        for (int e = lane; e < n; e += 32) cnt += (akey(z[e]) >= c);
        if (__reduce_add_sync(kFull, cnt) >= K) tau = c;
    }
    int above = 0, ties = 0;
    for (int e = lane; e < n; e += 32) {
        const uint32_t k = akey(z[e]);
        above += (k > tau);
        ties += (k == tau);
    }
    above = __reduce_add_sync(kFull, above);
    ties = __reduce_add_sync(kFull, ties);
    const int need = K - above;  // 1 <= need <= ties
    uint32_t cut;
    if (need == ties) {
        uint32_t m = 0;
        for (int e = lane; e < n; e += 32)
            if (akey(z[e]) == tau) m = max(m, id[e]);
        cut = __reduce_max_sync(kFull, m);
    } else {
        uint32_t v = 0;  // need-th smallest index among the ties
        for (int b = 31; b >= 0; --b) {
            const uint32_t c = v | (1u << b);
            int cnt = 0;
            for (int e = lane; e < n; e += 32) cnt += (akey(z[e]) == tau && id[e] < c);
            if (__reduce_add_sync(kFull, cnt) < need) v = c;
        }
        cut = v;
    }
    tau_key = tau;
    tau_idx = cut;
}

__device__ __forceinline__ bool keeps(float z, uint32_t id, uint32_t tau_key, uint32_t tau_idx) {
    const uint32_t k = akey(z);
    return k > tau_key || (k == tau_key && id <= tau_idx);
}

// In-place compaction of the entries of (z, id)[0..n) that satisfy
// keeps(); order is preserved. Returns the new length.
__device__ __forceinline__ int warp_compact_keep(float *z, uint32_t *id, int n, uint32_t tau_key,
                                                 uint32_t tau_idx) {
    const int lane = threadIdx.x & 31;
    int out = 0;
    for (int e0 = 0; e0 < n; e0 += 32) {
        const int e = e0 + lane;
        float zv = 0.f;
        uint32_t iv = 0;
        bool k = false;
        if (e < n) {
            zv = z[e];
            iv = id[e];
            k = keeps(zv, iv, tau_key, tau_idx);
        }
        const unsigned m = __ballot_sync(kFull, k);
        __syncwarp();
        if (k) {
            const int pos = out + __popc(m & ((1u << lane) - 1u));
            z[pos] = zv;
            id[pos] = iv;
        }
        out += __popc(m);
        __syncwarp();
    }
    return out;
}

// Composite order key: candidates compare by (key desc, idx asc). Entries
// marked invalid use key 0 and are never selected (valid keys are stored +1).
struct Cand {
    uint32_t key;  // |z| bits + 1, or 0 for "no candidate"
    uint32_t idx;
    float z;
};

__device__ __forceinline__ bool cand_before(const Cand &a, const Cand &b) {
    return a.key > b.key || (a.key == b.key && a.idx < b.idx);
}

__device__ __forceinline__ void cand_swap_if(Cand &a, Cand &b) {
    if (cand_before(b, a)) {
        const Cand t = a;
        a = b;
        b = t;
    }
}

// The B first of up to 128 candidates held 4 per lane (c[0..3]), by B
// rounds of a warp-wide tournament over the lanes' sorted heads. Writes the
// winners' (z, idx) to out_z / out_id (lane 0) in order; returns how many
// valid candidates were taken (<= B).
__device__ __forceinline__ int warp_tournament4(Cand (&c)[4], int B, float *out_z, uint32_t *out_id) {
    cand_swap_if(c[0], c[1]);
    cand_swap_if(c[2], c[3]);
    cand_swap_if(c[0], c[2]);
    cand_swap_if(c[1], c[3]);
    cand_swap_if(c[1], c[2]);
    int taken = 0;
    for (int r = 0; r < B; ++r) {
        const uint32_t m = __reduce_max_sync(kFull, c[0].key);
        if (m == 0) break;
        const uint32_t im = __reduce_min_sync(kFull, c[0].key == m ? c[0].idx : 0xffffffffu);
        if (c[0].key == m && c[0].idx == im) {
            out_z[r] = c[0].z;
            out_id[r] = c[0].idx;
            c[0] = c[1];
            c[1] = c[2];
            c[2] = c[3];
            c[3].key = 0;
        }
        ++taken;
    }
    __syncwarp();
    return taken;
}

}  // namespace dpb
