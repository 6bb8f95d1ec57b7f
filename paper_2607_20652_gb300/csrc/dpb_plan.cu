// dpb_plan.cu -- host-side plan builder: configuration resolution, the field
// GF(2^t), the seed matrix M and the generators of every level. Runs once per
// plan; nothing here is on the per-token path.
//
// Field arithmetic follows App. A.2 of the paper (polynomial basis modulo an
// irreducible p(z)); inverses use discrete log / antilog tables over a
// primitive element, which give the same unique inverse xi^{2^t-2} of Eq. 25.
// The seed-matrix row packing is App. A.4 Eq. 22 with the low t bits meeting
// coord(xi) and the next t bits meeting coord(xi^{-1}).
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "dpb_internal.h"

namespace dpb {

namespace {

thread_local char g_last_error[512] = "";

// ---- polynomials over GF(2), as bit masks (bit j = coefficient of z^j) ----

int pdeg(uint64_t a) { return a ? 63 - __builtin_clzll(a) : -1; }

uint64_t pmod(uint64_t a, uint64_t b) {
    const int db = pdeg(b);
    for (int da = pdeg(a); da >= db; da = pdeg(a)) a ^= b << (da - db);
    return a;
}

uint64_t pgcd(uint64_t a, uint64_t b) {
    while (b) {
        uint64_t r = pmod(a, b);
        a = b;
        b = r;
    }
    return a;
}

// (a * b) mod p for polynomials of degree < deg p <= 16.
uint64_t pmulmod(uint64_t a, uint64_t b, uint64_t p) {
    uint64_t r = 0;
    for (; b; b >>= 1, a <<= 1) {
        if (b & 1) r ^= a;
        if (a >> pdeg(p) & 1) a ^= p;  // keep a reduced as it is shifted
    }
    return pmod(r, p);
}

// Rabin's test: p of degree t is irreducible iff z^{2^t} = z (mod p) and
// gcd(z^{2^{t/q}} - z, p) = 1 for every prime q dividing t.
bool irreducible(int t, uint64_t p) {
    if (t < 1 || pdeg(p) != t) return false;
    auto z_pow_2k = [&](int k) {  // z^{2^k} mod p by k squarings
        uint64_t v = pmod(2, p);
        for (int i = 0; i < k; ++i) v = pmulmod(v, v, p);
        return v;
    };
    if (z_pow_2k(t) != pmod(2, p)) return false;
    for (int q = 2; q <= t; ++q) {
        bool prime = true;
        for (int f = 2; f * f <= q; ++f)
            if (q % f == 0) prime = false;
        if (!prime || t % q) continue;
        uint64_t g = pgcd(p, z_pow_2k(t / q) ^ pmod(2, p));
        if (pdeg(g) > 0) return false;
    }
    return true;
}

uint32_t default_poly(int t) {
    if (t == 10) return (1u << 10) | (1u << 3) | 1u;  // App. A.4, Eq. 24
    if (t == 11) return (1u << 11) | (1u << 2) | 1u;  // App. A.4, Eq. 24
    const uint32_t top = 1u << t;
    for (int a = 1; a < t; ++a)
        if (irreducible(t, top | (1u << a) | 1u)) return top | (1u << a) | 1u;
    uint32_t best = 0;
    for (int a = 3; a < t; ++a)
        for (int b = 2; b < a; ++b)
            for (int c = 1; c < b; ++c) {
                uint32_t p = top | (1u << a) | (1u << b) | (1u << c) | 1u;
                if (irreducible(t, p) && (best == 0 || p < best)) best = p;
            }
    return best;
}

// ---- the field GF(2^t) ----

struct Field {
    int t;
    uint32_t poly, q;
    std::vector<uint32_t> exp_, log_;

    uint32_t mul(uint32_t a, uint32_t b) const {  // shift-and-add with reduction
        uint32_t r = 0;
        while (b) {
            if (b & 1) r ^= a;
            b >>= 1;
            a <<= 1;
            if (a & q) a ^= poly;
        }
        return r;
    }

    // Find a primitive element and fill the antilog/log tables.
    bool init(int t_, uint32_t poly_) {
        t = t_;
        poly = poly_;
        q = 1u << t;
        exp_.assign(q, 0);
        log_.assign(q, 0);
        for (uint32_t g = 2; g < q; ++g) {
            uint32_t v = 1, n = 0;
            do {
                exp_[n++] = v;
                v = mul(v, g);
            } while (v != 1 && n < q);
            if (n == q - 1) {
                for (uint32_t i = 0; i < q - 1; ++i) log_[exp_[i]] = i;
                return true;
            }
        }
        return q == 2;  // GF(2): the only nonzero element is 1
    }

    uint32_t inv(uint32_t a) const {  // 0^{-1} = 0 by convention (App. A.3)
        if (a == 0) return 0;
        if (q == 2) return 1;
        return exp_[(q - 1 - log_[a]) % (q - 1)];
    }
};

uint64_t splitmix64(uint64_t &s) {
    s += 0x9E3779B97F4A7C15ULL;
    uint64_t z = s;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

int ceil_log2(int v) {
    int r = 0;
    while ((1 << r) < v) ++r;
    return r;
}

}  // namespace

void build_mma_tables(dpb_plan *p) {
    const dpb_config &c = p->cfg;
    bool ok = c.dtype == DPB_BF16 && c.d % 32 == 0 && c.d >= 32 && c.d <= 1024 && c.levels >= 2 &&
              c.select_mode == DPB_SELECT_GLOBAL && c.beam >= 1 && c.beam <= 16 && c.k >= c.beam && c.k <= 256;
    for (int l = 1; l < c.levels && ok; ++l) ok = c.children[l] == 16;
    // a difference + 1 below 2^bits[L-2] must fit the 28 key bits of a DD entry
    ok = ok && c.bits[c.levels - 2] <= 27;
    const int nblk = c.d / 32;
    // every level's fragments, the tables and the warps' lists share one block
    p->mma_encode = ok;
    if (ok && encode_mma_warps(p) == 0) p->mma_encode = ok = false;
    if (!ok) return;
    p->FRAG.assign((size_t)(c.levels - 1) * nblk * 256, 0u);
    auto sign_bf16 = [&](uint32_t g, int iota) -> uint32_t {
        return (__builtin_popcount(p->M[iota] & g) & 1) ? 0xBF80u : 0x3F80u;
    };
    for (int l = 1; l < c.levels; ++l)
        for (int m = 0; m < nblk; ++m)
            for (int lane = 0; lane < 32; ++lane)
                for (int w = 0; w < 8; ++w) {
                    const int chunk = w / 4, half = (w / 2) % 2, reg = w % 2;
                    const int n = 8 * half + lane / 4, q4 = lane % 4, pair = 2 * chunk + reg;
                    const uint32_t g = p->G[(size_t)l * DPB_MAX_CHILDREN + n];
                    const int ia = 32 * m + frag_coord(q4, pair, 0), ib = 32 * m + frag_coord(q4, pair, 1);
                    // chunk-major: a warp's 128-bit loads of one chunk read 512
                    // contiguous bytes (no bank conflict)
                    p->FRAG[((((size_t)(l - 1) * nblk + m) * 2 + chunk) * 32 + lane) * 4 + w % 4] =
                        sign_bf16(g, ia) | (sign_bf16(g, ib) << 16);
                }
    p->DD.assign((size_t)(c.levels - 1) * kDedupSlots, 0u);
    for (int l = 1; l < c.levels; ++l) {
        uint32_t *tab = &p->DD[(size_t)(l - 1) * kDedupSlots];
        const uint32_t *g = &p->G[(size_t)l * DPB_MAX_CHILDREN];
        // parents of level l lie below 2^bits[l-1], so only differences below
        // that bound can make two parents share a child
        const uint32_t bound = 1u << c.bits[l - 1];
        for (int j = 0; j < 16; ++j)
            for (int jj = 0; jj < 16; ++jj) {
                if (j == jj) continue;
                const uint32_t delta = g[j] ^ g[jj];
                if (delta >= bound) continue;
                uint32_t h = dedup_hash(delta);
                while (tab[h] != 0) h = (h + 1) & (kDedupSlots - 1);
                tab[h] = ((delta + 1) << 4) | (uint32_t)j;
            }
    }
}

dpb_status fail(dpb_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
    return s;
}

const char *last_error_message() { return g_last_error; }

dpb_status resolve_and_build(const dpb_config *in, const uint32_t *generators, dpb_plan *p) {
    dpb_config c = *in;
    if (c.d < 2 || c.d > 4096) return fail(DPB_ERR_UNSUPPORTED, "d=%d outside [2, 4096]", c.d);
    if (c.levels < 1 || c.levels > DPB_MAX_LEVELS)
        return fail(DPB_ERR_INVALID_ARG, "levels=%d outside [1, %d]", c.levels, DPB_MAX_LEVELS);
    const int r0 = ceil_log2(c.d);
    bool derive_bits = true;
    for (int l = 0; l < DPB_MAX_LEVELS; ++l)
        if (c.bits[l]) derive_bits = false;
    if (derive_bits) {
        if (c.levels == 1) {
            c.bits[0] = r0;
        } else {
            if (c.m_bits <= r0) return fail(DPB_ERR_INVALID_ARG, "m_bits=%d must exceed ceil(log2 d)=%d", c.m_bits, r0);
            for (int l = 0; l < c.levels; ++l) c.bits[l] = r0 + (l * (c.m_bits - r0)) / (c.levels - 1);
        }
    }
    if (c.bits[0] < r0) return fail(DPB_ERR_INVALID_ARG, "bits[0]=%d below ceil(log2 d)=%d", c.bits[0], r0);
    for (int l = 1; l < c.levels; ++l)
        if (c.bits[l] <= c.bits[l - 1]) return fail(DPB_ERR_INVALID_ARG, "bits must increase");
    for (int l = c.levels; l < DPB_MAX_LEVELS; ++l) c.bits[l] = 0;
    const int N = c.bits[c.levels - 1];
    c.m_bits = N;
    if (N > 31) return fail(DPB_ERR_UNSUPPORTED, "index space 2^%d exceeds 2^31", N);
    if (c.field_t == 0) c.field_t = std::max(r0, (N + 1) / 2);
    if (c.field_t < r0 || c.field_t > 16)
        return fail(DPB_ERR_UNSUPPORTED, "field_t=%d outside [ceil(log2 d), 16]", c.field_t);
    if (2 * c.field_t < N)
        return fail(DPB_ERR_INVALID_ARG, "2t=%d bits of M cannot address 2^%d indices", 2 * c.field_t, N);
    if (c.field_poly == 0) c.field_poly = default_poly(c.field_t);
    if (!irreducible(c.field_t, c.field_poly))
        return fail(DPB_ERR_INVALID_ARG, "field_poly 0x%x is not an irreducible polynomial of degree %d",
                    c.field_poly, c.field_t);
    c.children[0] = 0;
    for (int l = 1; l < c.levels; ++l) {
        if (c.children[l] < 1 || c.children[l] > DPB_MAX_CHILDREN)
            return fail(DPB_ERR_UNSUPPORTED, "children[%d]=%d outside [1, %d]", l, c.children[l], DPB_MAX_CHILDREN);
        const uint64_t avail = (1ull << c.bits[l]) - (1ull << c.bits[l - 1]);
        if ((uint64_t)c.children[l] > avail)
            return fail(DPB_ERR_INVALID_ARG, "level %d has only %llu valid generators", l, (unsigned long long)avail);
    }
    for (int l = c.levels; l < DPB_MAX_LEVELS; ++l) c.children[l] = 0;
    if (c.norm_match != 0 && c.norm_match != 1) return fail(DPB_ERR_INVALID_ARG, "norm_match must be 0 or 1");
    if (c.dtype != DPB_F32 && c.dtype != DPB_BF16) return fail(DPB_ERR_INVALID_ARG, "unknown dtype %d", c.dtype);
    if (c.select_mode == DPB_SELECT_GLOBAL) {
        if (c.beam < 1 || c.beam > 32) return fail(DPB_ERR_UNSUPPORTED, "beam=%d outside [1, 32]", c.beam);
        if (c.k < 1 || c.k > 256) return fail(DPB_ERR_UNSUPPORTED, "k=%d outside [1, 256]", c.k);
        if (c.k > c.d) return fail(DPB_ERR_INVALID_ARG, "k=%d exceeds d=%d", c.k, c.d);
        p->code_len = c.k;
    } else if (c.select_mode == DPB_SELECT_PER_LEVEL) {
        const dpb_status st = check_per_level(c);
        if (st != DPB_OK) return st;
        p->code_len = 0;
        for (int l = 0; l < c.levels; ++l) p->code_len += c.k_per_level[l];
    } else {
        return fail(DPB_ERR_INVALID_ARG, "unknown select_mode %d", c.select_mode);
    }

    // field and seed matrix
    Field F;
    if (!F.init(c.field_t, c.field_poly)) return fail(DPB_ERR_INVALID_ARG, "field construction failed");
    p->M.resize(c.d);
    for (int iota = 0; iota < c.d; ++iota)
        p->M[iota] = (uint32_t)iota | (F.inv((uint32_t)iota) << c.field_t);

    // generators
    p->G.assign((size_t)DPB_MAX_LEVELS * DPB_MAX_CHILDREN, 0u);
    for (int l = 1; l < c.levels; ++l) {
        uint32_t *row = &p->G[(size_t)l * DPB_MAX_CHILDREN];
        if (generators) {
            for (int j = 0; j < c.children[l]; ++j) {
                uint32_t g = generators[(size_t)l * DPB_MAX_CHILDREN + j];
                if ((g >> c.bits[l]) != 0 || (g >> c.bits[l - 1]) == 0)
                    return fail(DPB_ERR_INVALID_ARG, "generator %u of level %d breaks the level rule", g, l);
                for (int jj = 0; jj < j; ++jj)
                    if (row[jj] == g) return fail(DPB_ERR_INVALID_ARG, "generator %u repeats at level %d", g, l);
                row[j] = g;
            }
            continue;
        }
        uint64_t s = c.generator_seed ^ ((uint64_t)l * 0x9E3779B97F4A7C15ULL);
        int n = 0;
        while (n < c.children[l]) {
            const uint32_t g = (uint32_t)(splitmix64(s) >> (64 - c.bits[l]));
            if ((g >> c.bits[l - 1]) == 0) continue;
            bool dup = false;
            for (int m = 0; m < n; ++m) dup |= (row[m] == g);
            if (!dup) row[n++] = g;
        }
    }
    // high-half sign tables for the table-driven backward
    p->kvh = (c.field_t + 4) / 5;
    // at least two chunks: the kernels for t <= 10 read chunks 0 and 1
    p->VH.assign((size_t)std::max(p->kvh, 2) * 32 * 32, 0u);
    if (c.d <= 1024) {
        for (int k = 0; k < p->kvh; ++k)
            for (int q = 0; q < 32; ++q)
                for (int v = 0; v < 32; ++v) {
                    uint32_t w = 0;
                    const uint32_t mask = (uint32_t)v << (5 * k);
                    for (int l = 0; l < 32; ++l) {
                        const int iota = 32 * q + l;
                        if (iota >= c.d) continue;
                        const uint32_t kappa = p->M[iota] >> c.field_t;
                        w |= (uint32_t)(__builtin_popcount(kappa & mask) & 1) << l;
                    }
                    p->VH[((size_t)k * 32 + q) * 32 + v] = w;
                }
    }
    // the same words for every 32-coordinate block of d <= 2048, [chunk][block][v]
    if (c.d <= 2048) {
        const int nblk = (c.d + 31) / 32, nk = std::max(p->kvh, 2);
        p->VH2.assign((size_t)nk * nblk * 32, 0u);
        for (int k = 0; k < p->kvh; ++k)
            for (int q = 0; q < nblk; ++q)
                for (int v = 0; v < 32; ++v) {
                    uint32_t w = 0;
                    const uint32_t mask = (uint32_t)v << (5 * k);
                    for (int l = 0; l < 32; ++l) {
                        const int iota = 32 * q + l;
                        if (iota >= c.d) continue;
                        const uint32_t kappa = p->M[iota] >> c.field_t;
                        w |= (uint32_t)(__builtin_popcount(kappa & mask) & 1) << l;
                    }
                    p->VH2[((size_t)k * nblk + q) * 32 + v] = w;
                }
    }
    p->cfg = c;
    build_mma_tables(p);
    if (c.scoring == DPB_SCORING_COSET_WHT) {
        // the variant outside the paper: every level's 16 generators one coset
        // g0 ^ {0..15} (given by the caller), scored by a 16-point WHT
        if (!generators) return fail(DPB_ERR_INVALID_ARG, "coset scoring needs the caller's generators");
        if (!p->mma_encode || c.beam > 8)
            return fail(DPB_ERR_UNSUPPORTED,
                        "coset scoring needs global selection, bf16, beam <= 8, 16 children, d a multiple of 32 up to 1024");
        const int nblk = c.d / 32;
        p->COSET.assign((size_t)(c.levels - 1) * (nblk + 16), 0u);
        for (int l = 1; l < c.levels; ++l) {
            const uint32_t *g = &p->G[(size_t)l * DPB_MAX_CHILDREN];
            uint32_t *row = &p->COSET[(size_t)(l - 1) * (nblk + 16)];
            for (int j = 0; j < 16; ++j) {
                if ((g[j] ^ g[0]) > 15u)
                    return fail(DPB_ERR_INVALID_ARG, "level %d: generator %u is not in the coset of %u", l, g[j], g[0]);
                row[nblk + j] = g[j] ^ g[0];
            }
            for (int m = 0; m < nblk; ++m) {
                uint32_t w = 0;
                for (int i = 0; i < 32; ++i) w |= (uint32_t)(__builtin_popcount(p->M[32 * m + i] & g[0]) & 1) << i;
                row[m] = w;
            }
        }
    } else if (c.scoring != DPB_SCORING_CONTRACTION) {
        return fail(DPB_ERR_INVALID_ARG, "scoring=%d unknown", c.scoring);
    }
    if (c.select_mode == DPB_SELECT_PER_LEVEL) build_per_level_tables(p);
    p->t = c.field_t;
    p->poly = c.field_poly;
    p->m_mask = (N >= 32) ? 0xffffffffu : ((1u << N) - 1u);
    p->inv_sqrt_d = (float)(1.0 / std::sqrt((double)c.d));
    return DPB_OK;
}

}  // namespace dpb
