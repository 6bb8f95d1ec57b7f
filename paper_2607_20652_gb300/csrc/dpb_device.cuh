// dpb_device.cuh -- device helpers shared by the DPB kernels: dtype access,
// on-chip generation of parity signs, warp-level exact top-k selection and a
// warp bitonic sort. Everything here runs inside one warp.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

#include "../../include/dpb.h"

namespace dpb {

constexpr unsigned kFull = 0xffffffffu;

// ---- element access ---------------------------------------------------------

__device__ __forceinline__ float ld_elem(const float *p, int64_t i) { return p[i]; }
__device__ __forceinline__ float ld_elem(const __nv_bfloat16 *p, int64_t i) {
    return __bfloat162float(p[i]);
}
__device__ __forceinline__ void st_elem(float *p, int64_t i, float v) { p[i] = v; }
__device__ __forceinline__ void st_elem(__nv_bfloat16 *p, int64_t i, float v) {
    p[i] = __float2bfloat16_rn(v);
}

// ---- one warp over the d elements of a row ----------------------------------
//
// Rows of x, y, grad_y, grad_x against a float row `buf` in shared memory.
// With VEC the lane takes 4 consecutive elements at a time (8-byte bf16 or
// 16-byte fp32 accesses; the caller guarantees d % 4 == 0 and aligned rows),
// otherwise one element at a time.

__device__ __forceinline__ float4 ld4(const __nv_bfloat16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u), __uint_as_float(u.y << 16),
                       __uint_as_float(u.y & 0xffff0000u));
}
__device__ __forceinline__ float4 ld4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ void st4(__nv_bfloat16 *p, float4 v) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
    uint2 u;
    u.x = *reinterpret_cast<const uint32_t *>(&a);
    u.y = *reinterpret_cast<const uint32_t *>(&b);
    *reinterpret_cast<uint2 *>(p) = u;
}
__device__ __forceinline__ void st4(float *p, float4 v) { *reinterpret_cast<float4 *>(p) = v; }

template <bool VEC>
struct RowOps {
    // buf[i] = v
    __device__ __forceinline__ static void fill(float *buf, int d, float v) {
        const int lane = threadIdx.x & 31;
        if (VEC) {
            for (int i = 4 * lane; i < d; i += 128) *reinterpret_cast<float4 *>(buf + i) = make_float4(v, v, v, v);
        } else {
            for (int i = lane; i < d; i += 32) buf[i] = v;
        }
    }
    // sum over the row of row[i]^2 (this lane's share)
    template <typename T>
    __device__ __forceinline__ static float sumsq(const T *row, int d) {
        const int lane = threadIdx.x & 31;
        float s = 0.f;
        if (VEC) {
            for (int i = 4 * lane; i < d; i += 128) {
                const float4 v = ld4(row + i);
                s += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
            }
        } else {
            for (int i = lane; i < d; i += 32) {
                const float v = ld_elem(row, i);
                s += v * v;
            }
        }
        return s;
    }
    // buf[i] = c * row[i]
    template <typename T>
    __device__ __forceinline__ static void scale_in(float *buf, const T *row, int d, float c) {
        const int lane = threadIdx.x & 31;
        if (VEC) {
#pragma unroll 2
            for (int i = 4 * lane; i < d; i += 128) {
                const float4 v = ld4(row + i);
                *reinterpret_cast<float4 *>(buf + i) = make_float4(c * v.x, c * v.y, c * v.z, c * v.w);
            }
        } else {
            for (int i = lane; i < d; i += 32) buf[i] = c * ld_elem(row, i);
        }
    }
    // srr += buf[i]^2, sgr += row[i] buf[i] (this lane's share)
    template <typename T>
    __device__ __forceinline__ static void dots(const float *buf, const T *row, int d, float &srr, float &sgr) {
        const int lane = threadIdx.x & 31;
        if (VEC) {
            for (int i = 4 * lane; i < d; i += 128) {
                const float4 r = *reinterpret_cast<const float4 *>(buf + i), g = ld4(row + i);
                srr += r.x * r.x + r.y * r.y + r.z * r.z + r.w * r.w;
                sgr += g.x * r.x + g.y * r.y + g.z * r.z + g.w * r.w;
            }
        } else {
            for (int i = lane; i < d; i += 32) {
                const float r = buf[i], g = ld_elem(row, i);
                srr += r * r;
                sgr += g * r;
            }
        }
    }
    // buf[i] = r[i]; sxx += x[i]^2, srr += r[i]^2, sgr += g[i] r[i] (this
    // lane's share): the three rows in one sweep
    template <typename T>
    __device__ __forceinline__ static void rows3(float *buf, const T *x, const T *g, const float *r, int d,
                                                 float &sxx, float &srr, float &sgr) {
        const int lane = threadIdx.x & 31;
        if (VEC) {
#pragma unroll 2  // the rows' loads of two trips in flight together
            for (int i = 4 * lane; i < d; i += 128) {
                const float4 xv = ld4(x + i), gv = ld4(g + i);
                const float4 rv = *reinterpret_cast<const float4 *>(r + i);
                sxx += xv.x * xv.x + xv.y * xv.y + xv.z * xv.z + xv.w * xv.w;
                srr += rv.x * rv.x + rv.y * rv.y + rv.z * rv.z + rv.w * rv.w;
                sgr += gv.x * rv.x + gv.y * rv.y + gv.z * rv.z + gv.w * rv.w;
                *reinterpret_cast<float4 *>(buf + i) = rv;
            }
        } else {
            for (int i = lane; i < d; i += 32) {
                const float xv = ld_elem(x, i), gv = ld_elem(g, i), rv = r[i];
                sxx += xv * xv;
                srr += rv * rv;
                sgr += gv * rv;
                buf[i] = rv;
            }
        }
    }
    // buf[i] = c (row[i] - beta buf[i])
    template <typename T>
    __device__ __forceinline__ static void project(float *buf, const T *row, int d, float c, float beta) {
        const int lane = threadIdx.x & 31;
        if (VEC) {
#pragma unroll 2
            for (int i = 4 * lane; i < d; i += 128) {
                const float4 r = *reinterpret_cast<const float4 *>(buf + i), g = ld4(row + i);
                *reinterpret_cast<float4 *>(buf + i) =
                    make_float4(c * (g.x - beta * r.x), c * (g.y - beta * r.y), c * (g.z - beta * r.z),
                                c * (g.w - beta * r.w));
            }
        } else {
            for (int i = lane; i < d; i += 32) buf[i] = c * (ld_elem(row, i) - beta * buf[i]);
        }
    }
    // row[i] = c * buf[i]
    template <typename T>
    __device__ __forceinline__ static void store(T *row, const float *buf, int d, float c) {
        const int lane = threadIdx.x & 31;
        if (VEC) {
            for (int i = 4 * lane; i < d; i += 128) {
                const float4 r = *reinterpret_cast<const float4 *>(buf + i);
                st4(row + i, make_float4(c * r.x, c * r.y, c * r.z, c * r.w));
            }
        } else {
            for (int i = lane; i < d; i += 32) st_elem(row, i, c * buf[i]);
        }
    }
};

// ---- parity signs (App. A.4, Eq. 26-27) ------------------------------------

// Sign of coordinate iota of phi~_c in bit 31: parity(M[iota] AND c), so a
// float is multiplied by R(.) = (-1)^bit with one XOR.
__device__ __forceinline__ uint32_t sign31(uint32_t m_row, uint32_t c) {
    return static_cast<uint32_t>(__popc(m_row & c)) << 31;
}
__device__ __forceinline__ float flip(float v, uint32_t s31) {
    return __uint_as_float(__float_as_uint(v) ^ s31);
}

// ---- ordering keys ----------------------------------------------------------

// |z| as an unsigned key: for finite floats the bit pattern of |z| orders like
// the value. Candidates are ordered by (key descending, index ascending).
__device__ __forceinline__ uint32_t akey(float z) { return __float_as_uint(z) & 0x7fffffffu; }

__device__ __forceinline__ bool before(uint32_t ka, uint32_t ia, uint32_t kb, uint32_t ib) {
    return ka > kb || (ka == kb && ia < ib);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

// ---- exact top-K of a shared-memory list -------------------------------------

// Writes the K first entries of (z[0..n), id[0..n)) in (|z| desc, id asc)
// order to (oz, oid), unordered, and returns K (n < K keeps all n). The K-th
// key is found by bisection on its bits (counts reduced across the warp), then
// ties on that key are cut by index with a second bisection. Warp-collective.
__device__ __forceinline__ int warp_select(const float *z, const uint32_t *id, int n, int K, float *oz,
                           uint32_t *oid) {
    const int lane = threadIdx.x & 31;
    if (K > n) K = n;
    uint32_t tau = 0;  // largest key with count(key >= tau) >= K
    if (K < n) {
        for (int b = 30; b >= 0; --b) {
            const uint32_t c = tau | (1u << b);
            int cnt = 0;
            for (int e = lane; e < n; e += 32) cnt += (akey(z[e]) >= c);
            if (__reduce_add_sync(kFull, cnt) >= K) tau = c;
        }
    }
    int above = 0, ties = 0;
    for (int e = lane; e < n; e += 32) {
        const uint32_t k = akey(z[e]);
        above += (k > tau);
        ties += (k == tau);
    }
    above = __reduce_add_sync(kFull, above);
    ties = __reduce_add_sync(kFull, ties);
    const int need = K - above;
    uint32_t cut = 0xffffffffu;  // ties with id <= cut are kept
    if (K < n && need < ties) {
        // cut = need-th smallest id among the ties
        uint32_t v = 0;
        for (int b = 31; b >= 0; --b) {
            const uint32_t c = v | (1u << b);
            int cnt = 0;
            for (int e = lane; e < n; e += 32) cnt += (akey(z[e]) == tau && id[e] < c);
            if (__reduce_add_sync(kFull, cnt) < need) v = c;
        }
        cut = v;
    }
    int base = 0;
    for (int e0 = 0; e0 < n; e0 += 32) {
        const int e = e0 + lane;
        bool keep = false;
        if (e < n) {
            const uint32_t k = akey(z[e]);
            keep = (K >= n) || k > tau || (k == tau && id[e] <= cut);
        }
        const unsigned m = __ballot_sync(kFull, keep);
        if (keep) {
            const int pos = base + __popc(m & ((1u << lane) - 1u));
            oz[pos] = z[e];
            oid[pos] = id[e];
        }
        base += __popc(m);
    }
    __syncwarp();
    return K;
}

// ---- warp bitonic sort -------------------------------------------------------

// Sorts (z, id)[0..n) in place into (|z| desc, id asc) order. `cap` is a power
// of two >= n; slots n..cap-1 are filled with a sentinel that sorts last.
__device__ __forceinline__ void warp_sort(float *z, uint32_t *id, int n, int cap) {
    const int lane = threadIdx.x & 31;
    for (int e = n + lane; e < cap; e += 32) {
        z[e] = 0.f;
        id[e] = 0xffffffffu;
    }
    __syncwarp();
    for (int size = 2; size <= cap; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = lane; i < cap; i += 32) {
                const int j = i ^ stride;
                if (j > i) {
                    const bool up = (i & size) == 0;  // this run ascends in (before) order
                    const uint32_t ki = akey(z[i]), kj = akey(z[j]);
                    const bool swap = up ? before(kj, id[j], ki, id[i]) : before(ki, id[i], kj, id[j]);
                    if (swap) {
                        const float tz = z[i];
                        z[i] = z[j];
                        z[j] = tz;
                        const uint32_t ti = id[i];
                        id[i] = id[j];
                        id[j] = ti;
                    }
                }
            }
            __syncwarp();
        }
    }
}

__device__ __forceinline__ void set_status(int32_t *status, int32_t bit) {
    if (status) atomicOr(status, bit);
}

// ---- score standardisation (§2.2 "Score Standardization") -------------------------

// z = (s - mu_c) / sigma_c, computed as (s - mu_c) * r_c with r_c = 1 / sigma_c
// rounded to fp32, so that every path gives the same z for the same s. `tab`
// (nullable) holds the pairs (mu_c, r_c): one 8-byte load instead of one from
// each table. A sigma that is not a positive finite number (r_c outside
// (0, inf)) sets DPB_DEV_BAD_SIGMA when `status` is given.
// The table entries (mu_c, 1 / sigma_c) of feature c: the packed pair, or one
// load from each table. No side effect, so that callers can issue a batch of
// them before using any: z = (s - e.x) * e.y, and zbad(e.y) flags a sigma that
// is not a positive finite number.
__device__ __forceinline__ float2 ztab(uint32_t c, const float *mu, const float *sigma, const float2 *tab) {
    if (tab) return tab[c];
    return make_float2(mu[c], __frcp_rn(sigma[c]));
}
__device__ __forceinline__ bool zbad(float r) { return !(r > 0.f && r <= 3.402823466e38f); }

__device__ __forceinline__ float zscore(float s, uint32_t c, const float *mu, const float *sigma,
                                        const float2 *tab, int32_t *status) {
    float m, r;
    if (tab) {
        const float2 p = tab[c];
        m = p.x;
        r = p.y;
    } else {
        m = mu[c];
        r = __frcp_rn(sigma[c]);
    }
    if (status && !(r > 0.f && r <= 3.402823466e38f)) set_status(status, DPB_DEV_BAD_SIGMA);
    return (s - m) * r;
}

}  // namespace dpb
