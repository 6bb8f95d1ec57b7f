// dpb_encode_pl.cu -- the paper's per-level encoder (§2.2 and the per-level
// configuration table of App. G): level 0 keeps its top K_0 coordinates;
// level l scores the Delta_l children p ^ g_j of every index kept at level
// l-1 and keeps its top K_l distinct children; the code is every level's kept
// set, level by level, each in (|z| descending, index ascending) order.
//
// Child scoring (Eq. 6) runs on the tcgen05 tensor cores. A block of 8 warps
// owns 8 tokens. At level l its tensor-core rows are (token, parent slot):
// 16 slots per token (one M = 128 tile) when K_{l-1} <= 16, else 32 (two
// tiles); its Delta_l columns are the level's generators, so one tcgen05.mma
// of M = 128, N = Delta_l, K = 16 scores 128 x Delta_l children at once. Tile
// t's TMEM lane quarter q holds the rows of token q + 4 t (32 slots), or of
// tokens q and q + 4 (16 slots each), so that warp w reads its token's rows
// from its own quarter. K runs over d in chunks of 64 coordinates, double
// buffered:
//  - A (128 x 64 bf16) is built in shared memory by the block's threads,
//    each writing its row x (.) phi~_parent: the token's x pairs XOR the
//    parent's sign bits (App. A.4 Eq. 26 tables), in the K-major core-matrix
//    layout with the K order permuted so that K positions (2i, 2i+1) of a
//    32-coordinate block hold coordinates (i, i + 16), whose sign bits one
//    shift moves to the bf16 sign positions;
//  - B (Delta_l x 64 bf16, the generators' +-1 signs in the same order) is
//    one bulk copy of the plan's precomputed tile, issued by a tenth warp's
//    lane 0 (the producer) once the MMAs that last read its stage are done;
//  - a ninth warp's lane 0 issues the MMAs of a chunk once the 8 token
//    warps have arrived on the A stage's mbarrier and the generator tile has
//    landed, and commits them to an mbarrier that frees the chunk's buffers;
//    scores accumulate in TMEM. The token warps build the next A stages
//    meanwhile (two of two tiles, or four of one tile), so no warp both
//    builds A and waits to issue.
// Every mbarrier wait is bounded; a wait that gives up sets
// DPB_DEV_TIMEOUT and stops the block, which then waits (again bounded) for
// its bulk copies and MMAs still in flight and frees its TMEM.
//
// Selection of a level (one warp per token, lane = parent slot): each lane
// keeps the 4 largest of its row's group maxima (the largest key |z| of each
// 8 consecutive children; at level 0, of each 8 of the lane's coordinates
// lane + 32 j with consecutive j), the warp sorts the union and
// takes a threshold tau at rank K of its distinct keys. Each of those keys is
// a candidate's, so at least K distinct candidates reach tau, and with them
// the level's top K. Every candidate at or above tau is gathered (one pass
// with running ballot positions), sorted, and its repeated indices (two
// parents can share a child) are dropped; the first K remain.
#include <algorithm>
#include <atomic>
#include <type_traits>

#include "dpb_encode_mma.cuh"
#include "dpb_internal.h"

namespace dpb {

namespace {

constexpr int kTokens = 8;      // tokens per block, one per warp
constexpr int kThreads = (kTokens + 2) * 32;  // and a ninth warp, whose lane 0 issues the MMAs,
constexpr int kIssuer = kTokens * 32;         // and a tenth, whose lane 0 copies the generator tiles
constexpr int kProducer = (kTokens + 1) * 32;
constexpr int kRows = 32;       // tensor-core rows per token (parent slots)
constexpr int kChunk = 64;      // coordinates per K chunk
constexpr int kATile = 128 * kChunk * 2;  // one M = 128 tile of a chunk
constexpr int kSelCap = 256;    // gathered candidates per token and level (up to 8 per lane)
constexpr int kMaxK = 64;       // K_l per level
constexpr int kMaxStages = 4;   // generator-tile stages in flight
constexpr uint32_t kSpin = 1u << 20;  // default bound of the main loop's mbarrier waits, and of the drain
// at least this much shared memory per block, so that one block (holding all
// 512 TMEM columns) runs per SM
constexpr int kMinSmem = 120 * 1024;

struct Args {
    const __nv_bfloat16 *x;
    int64_t T;
    const float *mu, *sigma;
    const float2 *tab;  // packed (mu, 1 / sigma), nullable
    int32_t *idx;
    float *val, *xnorm;
    int32_t *status;
    const uint32_t *GT, *G, *VH2;
    int d, nblk, levels, t, kvh, code_len, dmax, nbs;
    int kl[DPB_MAX_LEVELS], delta[DPB_MAX_LEVELS], off[DPB_MAX_LEVELS];
    int64_t gt_off[DPB_MAX_LEVELS];
    float inv_sqrt_d;
    uint32_t spin;  // bound (tries) of the main loop's mbarrier waits
};

// ---- layout --------------------------------------------------------------------

constexpr int kSelBytes = 8 * kSelCap;  // a warp's gathered (z, index) pairs

struct Layout {
    int a, b, xw, vh, g, w5, par, mbar, total;
};

// The gathered candidates of the 8 warps share the generator-tile stages: a
// level's selection starts once its MMAs are done and before the next
// level's tiles are copied.
__host__ __device__ inline Layout layout(int d, int levels, int kvh, int dmax, int nbs) {
    const int nblk = d / 32;
    const int bbytes = nbs * dmax * 128 > kTokens * kSelBytes ? nbs * dmax * 128 : kTokens * kSelBytes;
    Layout l;
    l.a = 0;
    l.b = l.a + 2 * 2 * kATile;  // 2 stages x 2 tiles
    l.xw = l.b + bbytes;
    l.vh = l.xw + kTokens * nblk * 16 * 4;
    l.g = l.vh + kvh * nblk * 32 * 4;
    l.w5 = l.g + levels * 256 * 4;
    l.par = l.w5 + 32 * 4;
    l.mbar = l.par + kTokens * kRows * 4;
    l.total = l.mbar + (2 * kMaxStages + 6) * 8 + 16;
    return l;
}

// ---- PTX wrappers ----------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ bool mbar_wait(uint32_t mbar, uint32_t parity, uint32_t spin) {
    for (uint32_t i = 0; i < spin; ++i) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(mbar), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

// Shared-memory matrix descriptor: K-major, no swizzle, 16-byte core-matrix
// rows, 128 bytes between core matrices along K, 1024 between 8-row groups.
__device__ __forceinline__ uint64_t tile_desc(uint32_t saddr) {
    return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)(128 >> 4) << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46);
}

// Bulk copy of one generator tile (D rows x 128 bytes) into shared memory,
// completing on mbarrier `full`.
__device__ __forceinline__ void copy_b(void *dst, const uint32_t *src, int D, uint32_t full) {
    const uint32_t bytes = (uint32_t)D * 128u;
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(full), "r"(bytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(full)
                 : "memory");
}

// Issues the load of 32 consecutive 32-bit columns of this warp's 32 TMEM
// lanes (one lane per thread). The registers hold the data only after
// tmem_ld_wait on them.
__device__ __forceinline__ void tmem_ld32_issue(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
        "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
}

// Waits for this thread's TMEM loads. The registers of the load are tied in
// as read-write operands, so that no use of them is scheduled before the wait.
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&v)[32]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                   "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]),
                   "+r"(v[15]), "+r"(v[16]), "+r"(v[17]), "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]),
                   "+r"(v[22]), "+r"(v[23]), "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]),
                   "+r"(v[29]), "+r"(v[30]), "+r"(v[31])
                 :
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    tmem_ld32_issue(taddr, v);
    tmem_ld_wait(v);
}

// Stores 32 consecutive 32-bit columns of this warp's 32 TMEM lanes (one
// lane per thread) and waits for the stores.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,"
        "%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
        "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]),
        "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]),
        "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// ---- selection ---------------------------------------------------------------------

struct WarpBufs {
    uint32_t *par;   // [32] parents of the next level
    float *z;        // [kSelCap]
    uint32_t *id;    // [kSelCap]
};

// One compare-exchange stage (size, stride) of a warp bitonic sort,
// descending, of 32 R 64-bit words held R per lane (element lane * R + r).
template <int R>
__device__ __forceinline__ void sort_stage64(uint64_t (&v)[R], int size, int stride) {
    const int lane = threadIdx.x & 31;
    if (stride >= R) {
        const bool lower = (lane & (stride / R)) == 0;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const bool desc = (((lane * R + r) & size) == 0);
            const uint64_t o = __shfl_xor_sync(kFull, v[r], stride / R);
            const bool gt = v[r] > o;
            v[r] = (lower == desc) ? (gt ? v[r] : o) : (gt ? o : v[r]);
        }
    } else {
#pragma unroll
        for (int cs = 1; cs < R; cs <<= 1) {
            if (stride == cs) {
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int q = r ^ cs;
                    if (q > r) {
                        const bool desc = (((lane * R + r) & size) == 0);
                        const uint64_t hi = v[r] > v[q] ? v[r] : v[q], lo = v[r] > v[q] ? v[q] : v[r];
                        v[r] = desc ? hi : lo;
                        v[q] = desc ? lo : hi;
                    }
                }
            }
        }
    }
}

// Sorts the n (<= 32 R) gathered candidates as 64-bit words, drops repeated
// indices (equal candidates score equally, so copies sit side by side) and
// writes the first K to code columns [col, col + K) of row `tok` (and the
// parents of the next level). Returns the number of distinct candidates.
template <int R>
__device__ __forceinline__ int sort_keep(int n, int K, const WarpBufs &w, const Args &a, int64_t tok, int col,
                                         bool par_out, bool write) {
    const int lane = threadIdx.x & 31;
    uint64_t v[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int e = R * lane + r;
        v[r] = e < n ? mmaenc::cword(w.z[e], w.id[e]) : 0ull;
    }
#pragma unroll 1
    for (int size = 2; size <= 32 * R; size <<= 1)
#pragma unroll 1
        for (int stride = size / 2; stride > 0; stride >>= 1) sort_stage64<R>(v, size, stride);
    bool keep[R];
    uint32_t prev = __shfl_up_sync(kFull, mmaenc::cword_idx(v[R - 1]), 1);
    int kept = 0;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const uint32_t id = mmaenc::cword_idx(v[r]);
        keep[r] = v[r] != 0ull && ((r == 0 && lane == 0) || id != prev);
        prev = id;
        kept += keep[r];
    }
    int base = kept;  // exclusive prefix of kept entries over the lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(kFull, base, o);
        if (lane >= o) base += t;
    }
    const int distinct = __shfl_sync(kFull, base, 31);
    base -= kept;
    if (write) {
        if (par_out) w.par[lane] = 0u;
        __syncwarp();
#pragma unroll
        for (int r = 0; r < R; ++r) {
            if (keep[r] && base < K) {
                const uint32_t id = mmaenc::cword_idx(v[r]);
                a.idx[tok * a.code_len + col + base] = (int32_t)id;
                a.val[tok * a.code_len + col + base] = mmaenc::cword_z(v[r]);
                if (par_out && base < kRows) w.par[base] = id;
            }
            base += keep[r];
        }
    }
    __syncwarp();
    return distinct;
}

// Sorts the union of the lanes' R keys (each lane's already descending; 0 =
// empty) and ranks its distinct keys (copies of one child share a key):
// drank[r] = rank of key r among them, 0 for a repeat or an empty slot.
// Returns the number of distinct keys.
template <int R>
__device__ __forceinline__ int union_distinct(uint32_t (&v)[R], int (&drank)[R]) {
    const int lane = threadIdx.x & 31;
    mmaenc::warp_sort_desc_runs<R>(v);
    uint32_t prev = __shfl_up_sync(kFull, v[R - 1], 1);
    int cnt = 0;
    bool first[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
        first[r] = v[r] != 0u && ((r == 0 && lane == 0) || v[r] != prev);
        prev = v[r];
        cnt += first[r];
    }
    int base = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(kFull, base, o);
        if (lane >= o) base += t;
    }
    base -= cnt;
    int nd = 0;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        drank[r] = first[r] ? base + 1 : 0;
        base += first[r];
        nd = max(nd, drank[r]);
    }
    return (int)__reduce_max_sync(kFull, (uint32_t)nd);
}

// The union's distinct key of rank `target` (0 if none).
template <int R>
__device__ __forceinline__ uint32_t key_of_rank(const uint32_t (&v)[R], const int (&drank)[R], int target) {
    uint32_t mine = 0u;
#pragma unroll
    for (int r = 0; r < R; ++r)
        if (drank[r] == target) mine = v[r];
    return __reduce_max_sync(kFull, mine);
}

// The top K distinct candidates of one token, as explained in the header.
// `scan(f)` calls f(v, live, gend, index) for every candidate of this lane (the
// first nlive lanes hold candidates), in
// the same order each time and in step across the warp: v is its score before
// the factor `scale` (> 0; the score is z = v scale), gend marks the last
// candidate of a group (a group is live or not as a whole), and index() gives
// its feature index. Scaling is monotone, so a group's largest |z| is its
// largest |v| scaled once. Writes code columns [col, col + K) of row `tok`
// and, when `par_out`, the kept indices as the next level's parents. Returns
// the number of distinct candidates kept (< K only with the status bit set).
template <class Scan>
__device__ __forceinline__ int select_level(Scan scan, int nlive, float scale, int K, const WarpBufs &w,
                                            const Args &a, int64_t tok, int col, bool par_out) {
    const int lane = threadIdx.x & 31;
    uint32_t top[4];
    int nd = 0;  // distinct keys in the union
    // Group maxima first; when they hold fewer than K distinct keys (rows of
    // few children, or copies), every candidate's key instead.
    // each lane's 4 largest keys: of its group maxima, or (EVERY) of all its
    // candidates; the choice is made at compile time, out of the candidate loop
    auto lane_keys = [&](auto every) {
#pragma unroll
        for (int r = 0; r < 4; ++r) top[r] = 0u;
        float gm = -1.f;  // the largest |v| of the current group (-1: none live)
        scan([&](float v, bool live, bool gend, auto) {
            if (live) gm = fmaxf(gm, fabsf(v));
            if (gend || decltype(every)::value) {
                uint32_t c = gm >= 0.f ? akey(gm * scale) + 1u : 0u;
                gm = -1.f;
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const uint32_t hi = max(top[r], c);
                    c = min(top[r], c);
                    top[r] = hi;
                }
            }
        });
    };
    // the union of each lane's first R keys, sorted, and the distinct key of a
    // given rank in it: R = 2 when the nlive lanes that hold candidates give
    // at least 2 K keys that way, else R = 4
    uint32_t u2[2], u4[4];
    int dr2[2], dr4[4];
    const bool narrow = nlive >= K;
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {
        if (pass == 0)
            lane_keys(std::false_type{});
        else
            lane_keys(std::true_type{});
        if (narrow) {
            u2[0] = top[0];
            u2[1] = top[1];
            nd = union_distinct<2>(u2, dr2);
        } else {
#pragma unroll
            for (int r = 0; r < 4; ++r) u4[r] = top[r];
            nd = union_distinct<4>(u4, dr4);
        }
        if (nd >= K) break;
    }
    // tau = the union's distinct key of rank K: every key of the union is some
    // candidate's, so K distinct candidates reach it and the level's top K
    // distinct all do (the union's last distinct key when it holds fewer)
    const int target = min(K, nd);
    uint32_t tau = narrow ? key_of_rank<2>(u2, dr2, target) : key_of_rank<4>(u4, dr4, target);
    if (tau == 0u) tau = 1u;
    // key(z) + 1 >= tau exactly when |z| >= the float with bits tau - 1
    const float tf = __uint_as_float(tau - 1u);
    // gather every candidate at or above tau, warp-interleaved in scan order
    // (one pass: positions come from the running ballot counts)
    int n = 0;
    scan([&](float v, bool live, bool, auto index) {
        const float z = v * scale;
        const bool take = live && fabsf(z) >= tf;
        const unsigned mb = __ballot_sync(kFull, take);
        if (mb) {  // rare: most candidates fall short of tau
            const int pos = n + __popc(mb & ((1u << lane) - 1u));
            if (take && pos < kSelCap) {
                w.z[pos] = z;
                w.id[pos] = index();
            }
            n += __popc(mb);
        }
    });
    if (n > kSelCap) {
        set_status(a.status, DPB_DEV_SHORT_CODE);
        n = kSelCap;
    }
    __syncwarp();
    // the narrowest sort that holds them: 32, 64, 128 or 256 words
    const int distinct = n <= 32    ? sort_keep<1>(n, K, w, a, tok, col, par_out, true)
                         : n <= 64  ? sort_keep<2>(n, K, w, a, tok, col, par_out, true)
                         : n <= 128 ? sort_keep<4>(n, K, w, a, tok, col, par_out, true)
                                    : sort_keep<8>(n, K, w, a, tok, col, par_out, true);
    if (distinct < K) {
        set_status(a.status, DPB_DEV_SHORT_CODE);
        for (int e = distinct + lane; e < K; e += 32) {
            a.idx[tok * a.code_len + col + e] = 0;
            a.val[tok * a.code_len + col + e] = 0.f;
        }
    }
    __syncwarp();
    return distinct;
}

__device__ __forceinline__ float standardise(float s, uint32_t c, const Args &a, int32_t *status) {
    return a.mu ? zscore(s, c, a.mu, a.sigma, a.tab, status) : s;
}

// Standardised scores of one warp's TMEM rows, columns [cb, ce) (Delta = D
// children of parent p, live when ok): z = (s / sqrt(d) - mu_c) / sigma_c in
// place of s. Four columns' table loads are in flight at a time. Not inlined:
// its registers do not count against the kernel's, whose plain path runs
// without it.
__device__ __noinline__ void standardise_cols(const float *mu, const float *sigma, const float2 *tab,
                                              int32_t *status, float inv_sqrt_d, uint32_t taddr, int cb, int ce,
                                              int D, bool ok, uint32_t p, const uint32_t *gl) {
    bool bad = false;
    for (int c0 = cb; c0 < ce; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(taddr + c0, v);
#pragma unroll
        for (int h = 0; h < 32; h += 4) {
            float2 e[4];
#pragma unroll
            for (int j = 0; j < 4; ++j)
                e[j] = ok && c0 + h + j < D ? ztab(p ^ gl[c0 + h + j], mu, sigma, tab) : make_float2(0.f, 1.f);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                v[h + j] = __float_as_uint((__uint_as_float(v[h + j]) * inv_sqrt_d - e[j].x) * e[j].y);
                bad |= zbad(e[j].y);
            }
        }
        tmem_st32(taddr + c0, v);
    }
    if (bad) set_status(status, DPB_DEV_BAD_SIGMA);
}

// ---- the kernel ----------------------------------------------------------------------

__global__ void __launch_bounds__(kThreads, 1) encode_pl_kernel(Args a) {
    extern __shared__ __align__(1024) uint8_t smem[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = a.d, nblk = a.nblk, L = a.levels;
    const Layout lay = layout(d, L, a.kvh, a.dmax, a.nbs);
    uint8_t *sA = smem + lay.a;
    uint8_t *sB = smem + lay.b;
    uint32_t *xw = reinterpret_cast<uint32_t *>(smem + lay.xw);
    uint32_t *vh = reinterpret_cast<uint32_t *>(smem + lay.vh);
    uint32_t *gs = reinterpret_cast<uint32_t *>(smem + lay.g);
    uint32_t *w5 = reinterpret_cast<uint32_t *>(smem + lay.w5);
    // full_b[stages], mma_done[stages], a_full[2 + 4]
    uint64_t *mbar = reinterpret_cast<uint64_t *>(smem + lay.mbar);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + 2 * kMaxStages + 6);
    WarpBufs wb;
    wb.par = reinterpret_cast<uint32_t *>(smem + lay.par) + warp * kRows;
    wb.z = reinterpret_cast<float *>(sB + warp * kSelBytes);
    wb.id = reinterpret_cast<uint32_t *>(sB + warp * kSelBytes + 4 * kSelCap);
    for (int i = tid; i < a.kvh * nblk * 32; i += blockDim.x) vh[i] = a.VH2[i];
    for (int i = tid; i < L * 256; i += blockDim.x) gs[i] = a.G[(i >> 8) * DPB_MAX_CHILDREN + (i & 255)];
    if (tid < 32) {
        uint32_t word = 0;
        for (int l = 0; l < 32; ++l) word |= (uint32_t)(__popc(l & tid) & 1) << l;
        w5[tid] = word;
    }
    if (tid == 0) {
        for (int i = 0; i < 2 * kMaxStages; ++i)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(mbar + i)));
        for (int i = 0; i < 6; ++i)  // an A stage is built once each of the token warps arrives
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(mbar + 2 * kMaxStages + i)),
                         "r"(kTokens));
        asm volatile("fence.mbarrier_init.release.cluster;");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(smem_u32(tmem_slot)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;");
    const uint32_t tmem = *tmem_slot;
    // Chunk g (counted over every level and group) uses A stage g & 1 and
    // generator stage g % nbs; its copy completes full_b[g % nbs] and its MMAs'
    // commit mma_done[g % nbs], each the (g / nbs)-th time, so the parity of
    // that count names the phase to wait for. Waits never fall a phase behind:
    // a stage is refilled only after the MMAs that read it are seen done.
    const int nbs = a.nbs;
    const uint32_t mbar0 = smem_u32(mbar);
    auto full_b = [&](uint32_t g) { return mbar0 + 8u * (g % (uint32_t)nbs); };
    auto mma_done = [&](uint32_t g) { return mbar0 + 8u * (kMaxStages + g % (uint32_t)nbs); };
    auto phase = [&](uint32_t g) { return (g / (uint32_t)nbs) & 1u; };
    auto stage_b = [&](uint32_t g) { return sB + (g % (uint32_t)nbs) * a.dmax * 128; };
    // A stages: a level of two M = 128 tiles has two of 32 KB, a level of one
    // tile four of 16 KB (the same region; two of them with fewer than four
    // generator stages). Counting the chunks of each kind
    // of level over every level and group (ga), chunk ga of a two-tile level
    // uses stage and mbarrier a_full[ga & 1] and of a one-tile level stage
    // ga & 3 and a_full[2 + (ga & 3)], each the (ga / stages)-th time.
    uint32_t G = 0;  // chunks of the levels done so far (every thread)
    uint32_t GA2 = 0, GA4 = 0;  // chunks of two-tile and of one-tile levels done so far
    bool failed = false;
    // generator tiles are copied (by the producer) and consumed (by the issuer) in
    // chunk order: the copies of chunks [consumed, issued) are in flight; the
    // issuer has committed the MMAs of Gc chunks
    uint32_t issued = 0, consumed = 0, Gc = 0;
    bool tfail = false;  // a wait of this thread gave up
    auto issue_b = [&](uint32_t g, const uint32_t *src, int D) {
        copy_b(stage_b(g), src, D, full_b(g));
        issued = g + 1;
    };
    const uint32_t lo_mask = (1u << a.t) - 1u;
    const int64_t ngroups = (a.T + kTokens - 1) / kTokens;
    uint16_t *xh = reinterpret_cast<uint16_t *>(xw + warp * nblk * 16);

    for (int64_t grp = blockIdx.x; grp < ngroups && !failed; grp += gridDim.x) {
        const int64_t tok = grp * kTokens + warp;
        const bool live = warp < kTokens && tok < a.T;
        // ---- the row in the pair layout: word m*16 + i = (x[32m+i], x[32m+i+16]); |x|; level 0 ----
        if (live) {
            const uint4 *row = reinterpret_cast<const uint4 *>(a.x + tok * d);
            float ss = 0.f;
#pragma unroll 4  // the row's loads in flight together (4 chunks per lane at d = 1024)
            for (int ch = lane; ch < d / 8; ch += 32) {
                const uint4 v = row[ch];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const uint32_t bits = mmaenc::elem16(v, e);
                    const int cd = 8 * ch + e, m = cd >> 5, wl = cd & 31;
                    xh[(m * 16 + (wl & 15)) * 2 + (wl >> 4)] = (uint16_t)bits;
                    const float xf = __uint_as_float(bits << 16);
                    ss = fmaf(xf, xf, ss);
                }
            }
            ss = warp_sum(ss);
            if (lane == 0 && a.xnorm) a.xnorm[tok] = sqrtf(ss);
            __syncwarp();
            // a lane's coordinates lane + 32 j in groups of 8 consecutive j (d is
            // a multiple of 64, so every lane has the same count)
            auto scan0 = [&](auto f) {
                for (int i = lane; i < d; i += 32) {
                    const int m = i >> 5, wl = i & 31;
                    const float xv = __uint_as_float((uint32_t)xh[(m * 16 + (wl & 15)) * 2 + (wl >> 4)] << 16);
                    f(standardise(xv, (uint32_t)i, a, nullptr), true, (m & 7) == 7 || i + 32 >= d,
                      [&] { return (uint32_t)i; });
                }
            };
            if (a.mu)
                for (int i = lane; i < d; i += 32) standardise(0.f, (uint32_t)i, a, a.status);
            select_level(scan0, 32, 1.f, a.kl[0], wb, a, tok, a.off[0], L > 1);  // d >= 64: every lane holds 2+
        } else if (warp < kTokens) {
            wb.par[lane] = 0u;
            __syncwarp();
        }
        __syncthreads();

        for (int l = 1; l < L && !failed; ++l) {
            const int P = a.kl[l - 1], D = a.delta[l], nch = d / kChunk;
            const int pp = P <= 16 ? 16 : 32, ntiles = pp / 16;  // slots per token, M = 128 tiles
            // this thread builds block half hb of row rr of each tile
            const int rr = tid & 127, hb = tid >> 7;
            // A row that is no live parent (a slot past K_{l-1}, a token past T)
            // takes parent 0 and whatever x its buffer holds: the selection
            // reads only live rows, and an MMA row depends on its own A row only
            uint32_t iw5[2], iu[2], ihv[2][4];
            const uint32_t *ixt[2];
#pragma unroll
            for (int tt = 0; tt < 2; ++tt) {
                const int q = rr >> 5, jj = rr & 31;
                const int tokw = pp == 32 ? q + 4 * tt : q + 4 * (jj >> 4);
                const int slot = pp == 32 ? jj : jj & 15;
                const bool ok = tt < ntiles && grp * kTokens + tokw < a.T && slot < P;
                const uint32_t *par = reinterpret_cast<const uint32_t *>(smem + lay.par) + tokw * kRows;
                const uint32_t pv = ok ? par[slot] : 0u;
                iw5[tt] = w5[pv & 31u];
                iu[tt] = (pv & lo_mask) >> 5;
#pragma unroll
                for (int k = 0; k < 4; ++k) ihv[tt][k] = (pv >> min(a.t + 5 * k, 31)) & 31u;
                ixt[tt] = xw + tokw * nblk * 16;
            }
            const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(D >> 3) << 17) | (8u << 24);
            const uint32_t *gt = a.GT + a.gt_off[l];
            const uint32_t G0 = G;
            // four A stages of one tile; the builders then wait for chunk c - 4's
            // MMAs, on the mbarrier of generator stage (c - 4) % nbs, which no
            // later chunk before c reuses only when nbs >= 4
            const bool a4 = ntiles == 1 && nbs >= 4;
            const int na = a4 ? 4 : 2;
            const uint32_t GA0 = a4 ? GA4 : GA2;
            auto a_stage = [&](int c) {
                const uint32_t ga = GA0 + (uint32_t)c;
                return a4 ? sA + (ga & 3u) * kATile : sA + (ga & 1u) * 2 * kATile;
            };
            auto a_full = [&](int c) {
                const uint32_t ga = GA0 + (uint32_t)c;
                return mbar0 + 8u * (2 * kMaxStages + (a4 ? 2u + (ga & 3u) : (ga & 1u)));
            };
            auto a_phase = [&](int c) {
                const uint32_t ga = GA0 + (uint32_t)c;
                return a4 ? (ga >> 2) & 1u : (ga >> 1) & 1u;
            };
            bool bfail = false;  // a builder's wait gave up
            if (tid == kProducer) {
                // ---- the producer: the level's first nbs tiles at its start (every
                // earlier MMA is done, so every stage is free), then, once chunk
                // c - 2's MMAs are done, the tile of chunk c + nbs - 2 into the stage
                // they read
                for (int c = 0; c < min(nbs, nch); ++c) issue_b(G0 + c, gt + (int64_t)c * D * 32, D);
                for (int c = 2; c + nbs - 2 < nch; ++c) {
                    if (!mbar_wait(mma_done(G0 + c - 2), phase(G0 + c - 2), a.spin)) {
                        set_status(a.status, DPB_DEV_TIMEOUT);
                        tfail = true;
                        break;
                    }
                    const int next = c + nbs - 2;
                    issue_b(G0 + next, gt + (int64_t)next * D * 32, D);
                }
            } else if (tid == kIssuer) {
                // ---- the issuer: for each chunk, once its A stage is built and
                // its generator tile has landed, the MMAs and their commit
                for (int c = 0; c < nch; ++c) {
                    const uint32_t g = G0 + c;
                    if (!mbar_wait(a_full(c), a_phase(c), a.spin) || !mbar_wait(full_b(g), phase(g), a.spin)) {
                        set_status(a.status, DPB_DEV_TIMEOUT);
                        tfail = true;
                        break;
                    }
                    consumed = g + 1;
                    asm volatile("tcgen05.fence::after_thread_sync;");
                    const uint32_t bb = smem_u32(stage_b(g));
                    const uint8_t *As = a_stage(c);
                    for (int tt = 0; tt < ntiles; ++tt) {
                        const uint32_t ab = smem_u32(As + tt * kATile);
#pragma unroll
                        for (int k = 0; k < kChunk / 16; ++k) {
                            const uint32_t acc = (c > 0 || k > 0) ? 1u : 0u;
                            asm volatile(
                                "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                                "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem + 256 * tt),
                                "l"(tile_desc(ab + 256 * k)), "l"(tile_desc(bb + 256 * k)), "r"(idesc), "r"(acc));
                        }
                    }
                    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                        mma_done(g)));
                    Gc = g + 1;
                }
            } else if (tid < kIssuer) {
                // ---- the token warps build A: chunk c's stage is free once the
                // MMAs of chunk c - na are done (a stage of an earlier level is free)
                for (int c = 0; c < nch; ++c) {
                    const uint32_t g = G0 + c;
                    if (c >= na && !mbar_wait(mma_done(g - na), phase(g - na), a.spin)) {
                        bfail = true;
                        break;
                    }
                    uint8_t *As = a_stage(c);
#pragma unroll
                    for (int tt = 0; tt < 2; ++tt) {
                        if (tt < ntiles) {
                            const int m = 2 * c + hb;
                            uint32_t sw = iw5[tt] ^ (0u - (uint32_t)(__popc((uint32_t)m & iu[tt]) & 1));
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                if (k < a.kvh) sw ^= vh[(k * nblk + m) * 32 + ihv[tt][k]];
                            const uint4 *xs = reinterpret_cast<const uint4 *>(ixt[tt] + m * 16);
                            uint8_t *At = As + tt * kATile;
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const uint4 xv = xs[q];
                                const int sh = 15 - 4 * q;
                                uint4 av;
                                av.x = xv.x ^ ((sw << sh) & 0x80008000u);
                                av.y = xv.y ^ ((sw << (sh - 1)) & 0x80008000u);
                                av.z = xv.z ^ ((sw << (sh - 2)) & 0x80008000u);
                                av.w = xv.w ^ ((sw << (sh - 3)) & 0x80008000u);
                                *reinterpret_cast<uint4 *>(At + (rr >> 3) * 1024 + (4 * hb + q) * 128 + (rr & 7) * 16) =
                                    av;
                            }
                        }
                    }
                    // this thread's stores, then the warp's, are seen by the tensor
                    // cores once the issuer has seen the warp's arrival
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a_full(c)) : "memory");
                }
            }
            {
                // the last commit covers every MMA of the level
                const uint32_t gl1 = G0 + nch - 1;
                const bool ok = !bfail && !tfail && mbar_wait(mma_done(gl1), phase(gl1), a.spin);
                if (__syncthreads_or(!ok)) {
                    failed = true;
                    break;
                }
            }
            G = G0 + nch;
            if (a4)
                GA4 += nch;
            else
                GA2 += nch;
            asm volatile("tcgen05.fence::after_thread_sync;");
            const uint32_t *gl = gs + l * 256;
            // ---- standardised scores, once per candidate (§2.2): z replaces s in
            // TMEM, so the selection's three passes gather no tables. Warp w
            // takes quarter w % 4 (all 32 rows; with 16 slots a quarter holds
            // tokens q and q + 4) of tile w / 4, or with one tile half w / 4 of
            // the columns: all eight warps keep table loads in flight.
            if (a.mu) {
                if (warp < kTokens) {
                    const int q = warp & 3, tile = ntiles == 2 ? warp >> 2 : 0;
                    const int half = ((D + 31) / 32 + 1) / 2 * 32;  // whole 32-column loads
                    const int cb = ntiles == 2 ? 0 : (warp >> 2) * half, ce = ntiles == 2 ? D : min(D, cb + half);
                    const int tokw = pp == 32 ? q + 4 * tile : q + 4 * (lane >> 4);
                    const int slot = pp == 32 ? lane : lane & 15;
                    const bool ok = grp * kTokens + tokw < a.T && slot < P;
                    const uint32_t p = ok ? reinterpret_cast<const uint32_t *>(smem + lay.par)[tokw * kRows + slot] : 0u;
                    const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + 256u * tile;
                    standardise_cols(a.mu, a.sigma, a.tab, a.status, a.inv_sqrt_d, taddr, cb, ce, D, ok, p, gl);
                }
                asm volatile("tcgen05.fence::before_thread_sync;");
                __syncthreads();
                asm volatile("tcgen05.fence::after_thread_sync;");
            }
            // ---- the level's selection, one warp per token ----
            if (live) {
                // this warp's rows: tile (warp / 4 when 32 slots), quarter warp % 4,
                // lanes [base, base + pp) of it
                const int tile = pp == 32 ? warp >> 2 : 0, base = pp == 16 ? 16 * (warp >> 2) : 0;
                const uint32_t taddr = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + 256u * tile;
                const int slot = lane - base;
                const bool rv = slot >= 0 && slot < pp && slot < P;
                const uint32_t p = rv ? wb.par[slot] : 0u;
                const float scale = a.mu ? 1.f : a.inv_sqrt_d;  // TMEM holds z, or s sqrt(d)
                auto scanl = [&](auto f) {
                    for (int c0 = 0; c0 < D; c0 += 32) {
                        uint32_t v[32];
                        tmem_ld32(taddr + c0, v);
                        // D is a multiple of 16: columns c0 + 16 .. c0 + 31 exist as a
                        // whole or not at all, and a group of 8 is live as a whole
                        const bool hi = rv && c0 + 32 <= D;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            f(__uint_as_float(v[j]), j < 16 ? rv : hi, (j & 7) == 7, [&] { return p ^ gl[c0 + j]; });
                    }
                };
                select_level(scanl, P, scale, a.kl[l], wb, a, tok, a.off[l], l + 1 < L);
            }
            asm volatile("tcgen05.fence::before_thread_sync;");
            __syncthreads();
        }
    }
    if (failed) set_status(a.status, DPB_DEV_TIMEOUT);
    // drain (bounded, with the default bound): every generator-tile copy still
    // in flight lands, and the last commit (which covers every MMA issued)
    // arrives, before the block frees its TMEM and its shared memory. The
    // issuer's counts reach the producer through shared memory (failed is the
    // block's, so every thread is here)
    if (failed) {
        if (tid == kIssuer) {
            tmem_slot[1] = consumed;
            tmem_slot[2] = Gc;
        }
        __syncthreads();
        if (tid == kProducer) {
            for (uint32_t g = tmem_slot[1]; g < issued; ++g) mbar_wait(full_b(g), phase(g), kSpin);
            const uint32_t gc = tmem_slot[2];
            if (gc > 0) mbar_wait(mma_done(gc - 1), phase(gc - 1), kSpin);
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;");
    __syncthreads();
    if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
}

}  // namespace

// ---- host side ----------------------------------------------------------------------

dpb_status check_per_level(const dpb_config &c) {
    if (c.dtype != DPB_BF16) return fail(DPB_ERR_UNSUPPORTED, "per-level selection needs bf16 rows");
    if (c.d % kChunk != 0 || c.d < kChunk || c.d > 2048)
        return fail(DPB_ERR_UNSUPPORTED, "per-level selection needs d a multiple of 64 in [64, 2048] (d=%d)", c.d);
    int prev = 0;
    for (int l = 0; l < c.levels; ++l) {
        const int K = c.k_per_level[l];
        if (K < 1 || K > kMaxK) return fail(DPB_ERR_UNSUPPORTED, "k_per_level[%d]=%d outside [1, %d]", l, K, kMaxK);
        if (l == 0 && K > c.d) return fail(DPB_ERR_INVALID_ARG, "k_per_level[0]=%d exceeds d=%d", K, c.d);
        if (l >= 1) {
            const int D = c.children[l];
            if (D % 16 != 0 || D < 16 || D > 256)
                return fail(DPB_ERR_UNSUPPORTED, "per-level selection needs children[%d] a multiple of 16 in [16, 256]",
                            l);
            if (prev > kRows)
                return fail(DPB_ERR_UNSUPPORTED, "k_per_level[%d]=%d parents exceed %d", l - 1, prev, kRows);
            if (K > prev * D) return fail(DPB_ERR_INVALID_ARG, "k_per_level[%d]=%d exceeds its %d candidates", l, K, prev * D);
        }
        prev = K;
    }
    return DPB_OK;
}

void build_per_level_tables(dpb_plan *p) {
    const dpb_config &c = p->cfg;
    const int nch = c.d / kChunk;
    auto sign = [&](uint32_t g, int iota) -> uint32_t {
        return (__builtin_popcount(p->M[iota] & g) & 1) ? 0xBF80u : 0x3F80u;
    };
    // generator tiles: K position kk = 32 b + 2 i + h of chunk ch holds coordinate 32 (2 ch + b) + i + 16 h
    std::vector<uint16_t> gt;
    for (int l = 0; l < DPB_MAX_LEVELS; ++l) p->gt_off[l] = 0;
    for (int l = 1; l < c.levels; ++l) {
        const int D = c.children[l];
        p->gt_off[l] = (int64_t)gt.size() / 2;
        const size_t base = gt.size();
        gt.resize(base + (size_t)nch * D * kChunk, 0);
        const uint32_t *g = &p->G[(size_t)l * DPB_MAX_CHILDREN];
        for (int ch = 0; ch < nch; ++ch)
            for (int n = 0; n < D; ++n)
                for (int kk = 0; kk < kChunk; ++kk) {
                    const int b = kk / 32, i = (kk % 32) / 2, h = kk % 2;
                    const int iota = 32 * (2 * ch + b) + i + 16 * h;
                    const size_t byte = (size_t)(n / 8) * 1024 + (size_t)(kk / 8) * 128 + (n % 8) * 16 + (kk % 8) * 2;
                    gt[base + (size_t)ch * D * kChunk + byte / 2] = (uint16_t)sign(g[n], iota);
                }
    }
    p->GT.assign(gt.size() / 2, 0u);
    for (size_t w = 0; w < p->GT.size(); ++w) p->GT[w] = (uint32_t)gt[2 * w] | ((uint32_t)gt[2 * w + 1] << 16);
    // (VH2, the inverse-coordinate sign words per block, is built with the plan)
}

namespace {

// Bound of the main loop's mbarrier waits for the launches that follow (-1:
// the default kSpin); set by dpb_debug_set_wait_limit.
std::atomic<int32_t> g_wait_limit{-1};

// Generator-tile stages: as many as fit (at least 2).
int pl_stages(const dpb_config &c, int kvh, int dmax) {
    for (int nbs = kMaxStages; nbs > 2; --nbs)
        if ((size_t)layout(c.d, c.levels, kvh, dmax, nbs).total <= kMaxSmemPerBlock) return nbs;
    return 2;
}

int pl_dmax(const dpb_config &c) {
    int dmax = 16;
    for (int l = 1; l < c.levels; ++l) dmax = std::max(dmax, c.children[l]);
    return dmax;
}

}  // namespace

size_t encode_pl_smem(const dpb_plan *p) {
    const dpb_config &c = p->cfg;
    const int dmax = pl_dmax(c), kvh = std::max(1, (c.field_t + 4) / 5);
    return (size_t)std::max(layout(c.d, c.levels, kvh, dmax, pl_stages(c, kvh, dmax)).total, kMinSmem);
}

cudaError_t launch_encode_pl(const dpb_plan *p, const void *x, int64_t T, const float *mu, const float *sigma,
                             const float2 *tab, int32_t *idx, float *val, float *xnorm, int32_t *status,
                             cudaStream_t stream) {
    const dpb_config &c = p->cfg;
    Args a{};
    a.x = static_cast<const __nv_bfloat16 *>(x);
    a.T = T;
    a.mu = mu;
    a.sigma = sigma;
    a.tab = tab;
    a.idx = idx;
    a.val = val;
    a.xnorm = xnorm;
    a.status = status;
    a.GT = p->dGT;
    a.G = p->dG;
    a.VH2 = p->dVH2;
    a.d = c.d;
    a.nblk = c.d / 32;
    a.levels = c.levels;
    a.t = c.field_t;
    a.kvh = std::max(1, (c.field_t + 4) / 5);
    a.code_len = p->code_len;
    a.dmax = 16;
    int off = 0;
    for (int l = 0; l < c.levels; ++l) {
        a.kl[l] = c.k_per_level[l];
        a.delta[l] = l ? c.children[l] : 0;
        a.off[l] = off;
        off += c.k_per_level[l];
        a.gt_off[l] = p->gt_off[l];
        if (l) a.dmax = std::max(a.dmax, c.children[l]);
    }
    a.inv_sqrt_d = p->inv_sqrt_d;
    a.nbs = pl_stages(c, a.kvh, a.dmax);
    const int32_t lim = g_wait_limit.load(std::memory_order_relaxed);
    a.spin = lim < 0 ? kSpin : (uint32_t)lim;
    const size_t smem = encode_pl_smem(p);
    const cudaError_t e = allow_smem((const void *)encode_pl_kernel, smem);
    if (e != cudaSuccess) return e;
    const int64_t groups = (T + kTokens - 1) / kTokens;
    const int grid = (int)std::min<int64_t>(groups, (int64_t)std::max(p->sms, 1));
    encode_pl_kernel<<<grid, kThreads, smem, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace dpb

extern "C" dpb_status dpb_debug_set_wait_limit(int32_t tries) {
    if (tries < -1) return dpb::fail(DPB_ERR_INVALID_ARG, "tries must be -1 (default) or >= 0");
    dpb::g_wait_limit.store(tries, std::memory_order_relaxed);
    return DPB_OK;
}
