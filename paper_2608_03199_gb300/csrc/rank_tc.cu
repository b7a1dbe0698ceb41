// rank_tc.cu -- centroid ranking on the tcgen05 tensor cores (Sec. 2.3,
// Sec. 4.1: P_i = the nprobe centroids with the largest inner product with
// q_i, best first, equal scores by lower centroid id), for any nlist, with no
// score table and one exact contraction pass.
//
//   k_rank_screen  (nlist > 2,048, bulk pipeline) the first pass: one fp16
//              product of the hi halves per score; the epilogue writes the
//              maximum of each group of 64 (or 32) centroids.  Tiles of two
//              sub-tiles of 128 queries share every B stage.
//   k_rank_threshold  one warp per query: the nprobe-th largest group maximum
//              less the proven error bounds of both passes, a starting
//              threshold that at least nprobe centroids reach.
//   k_rank_bulk / k_rank_tc  the exact contraction (tc_bulk.cuh with the
//              centroids' tensor-core layout, else the converter pipeline of
//              tc_pipeline.cuh) against one range of centroids (B rows, 128
//              per chunk, in increasing id order).  Each epilogue thread owns
//              one query and appends the scores that reach its threshold to
//              the query's list: the starting threshold of the first pass
//              (two sub-tiles per tile where A fits tensor memory twice), or,
//              without a first pass, a running threshold from a 256-bin
//              histogram of the scores it has kept (shared memory) -- the
//              lower edge of the highest bin such that at least nprobe kept
//              scores lie in it or above.  A score below either threshold has
//              nprobe larger ones, so it cannot be among the nprobe best.  Up
//              to 2,048 centroids every score is kept (ids implicit).
//   k_rank_final / k_rank_dense_final  one warp per query: the candidates of
//              its ranges that reach their final thresholds, the exact nprobe
//              best of them by (score desc, id asc), sorted.  The lists are in
//              id order, so among equal scores the first taken are the lowest
//              ids.
// A query whose list overflowed (many equal scores, or an adversarial order)
// is finished by the exact FP32 ranking of rank_kernel.cu.
#include <cmath>
#include <vector>

#include "tc_bulk.cuh"
#include "tc_pipeline.cuh"

namespace sieve {

// selection: monotone map of fp32 to uint32 (larger float -> larger key); -0
// is mapped as +0 so that equal scores have equal keys
__device__ __forceinline__ uint32_t order_key(float s) {
    const uint32_t u = __float_as_uint(s + 0.f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// the inverse of order_key
__device__ __forceinline__ float key_score(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Running-threshold histogram: 256 bins of width 1/128 over scores in
// [-1, 1); scores outside fall into the end bins.  In raw accumulator units
// (scores x 2^16) a bin is 512 wide, so bin and edge are exact.
constexpr int kRankBins = 256;
constexpr int kRankBinStride = 260;   // bytes per query: 4-byte words offset by one bank per slot
constexpr size_t kRankEpiBytes = (size_t)tcp::kM * kRankBinStride;

__device__ __forceinline__ int rank_bin(float raw) {
    const float t = fminf(fmaxf(raw * (1.f / 512.f), -129.f), 128.f);
    const int b = __float2int_rd(t) + kRankBins / 2;
    return b < 0 ? 0 : (b > kRankBins - 1 ? kRankBins - 1 : b);
}

// lower edge of a bin in raw units; bin 0 takes everything
__device__ __forceinline__ float rank_edge_raw(int b) {
    return b == 0 ? -__int_as_float(0x7f800000) : (float)(b - kRankBins / 2) * 512.f;
}

// What the ranking contraction's epilogue does with a query's scores.
constexpr int kRankGroupMax = 0;   // the maximum of each group of `group` centroids
constexpr int kRankStream = 1;     // the scores that reach the running threshold
constexpr int kRankDense = 2;      // every score (ids implicit: the list position)
constexpr int kRankStreamInit = 3; // the scores that reach a given starting threshold (no histogram)

struct RankArgs {
    const float *Q;
    int64_t nq;
    const float *C;
    int64_t nlist;
    int d;
    int *status;     // nullable: where a bounded wait that gives up is reported
    const unsigned char *tc_cent;   // tensor-core layout of the centroids (bulk path)
    int nprobe;
    int nranges;     // centroid ranges per query tile
    int64_t range_len;   // centroids per range, a multiple of 128
    int cap;         // list slots per (query, range)
    float *list_s;   // [nq][nranges][cap] candidate scores, in id order
    int32_t *list_i; //                    and their centroid ids (not kRankDense)
    int *list_n;     // [nq][nranges] candidates offered (above cap: the list overflowed)
    float *list_edge;   // [nq][nranges] the final threshold score (-inf: none)
    const float *init_edge;   // kRankStream, nullable: [nq] starting threshold (score units)
    float *gmax;     // kRankGroupMax: [nq][gld] group maxima (score units)
    int64_t gld;
    int group;       // kRankGroupMax: centroids per group, 32 or 64
};

__device__ int g_rank_status_sink;

// kSubT sub-tiles of 128 queries per tile (tc_bulk.cuh); two only in modes
// that keep nothing in shared memory
template <int kMode, int kSubT = 1>
struct RankModeT {
    using Args = RankArgs;
    static constexpr int kN = 128;
    static constexpr int kSub = kSubT;
    static constexpr int kRows = kSubT * tcp::kM;   // queries per tile
    static_assert(kSubT == 1 || kMode == kRankGroupMax || kMode == kRankStreamInit,
                  "two sub-tiles: no shared-memory state");
    struct Tile {
        int64_t q0;    // first query
        int ni;
        int64_t c0;    // first centroid of the tile's range
        int64_t nb;    // centroids in the range
    };
    __device__ static int num_tiles(const Args &a) { return (int)ceil_div(a.nq, kRows) * a.nranges; }
    // every tile costs about the same: a static stride over the blocks
    __device__ static int *tile_counter(const Args &) { return nullptr; }
    __device__ static int d(const Args &a) { return a.d; }
    __device__ static int *status(const Args &a) { return a.status ? a.status : &g_rank_status_sink; }
    __device__ static Tile tile(const Args &a, int t) {
        Tile T;
        T.q0 = (int64_t)(t / a.nranges) * kRows;
        T.ni = (int)(a.nq - T.q0 < kRows ? a.nq - T.q0 : kRows);
        T.c0 = (int64_t)(t % a.nranges) * a.range_len;
        T.nb = a.nlist - T.c0 < a.range_len ? a.nlist - T.c0 : a.range_len;
        return T;
    }
    __device__ static const float *a_row(const Args &a, const Tile &T, int i) {
        return i < T.ni ? a.Q + (T.q0 + i) * a.d : nullptr;
    }
    __device__ static const float *b_row(const Args &a, const Tile &T, int64_t r) {
        return r < T.nb ? a.C + (T.c0 + r) * a.d : nullptr;
    }
    __device__ static const unsigned char *b_block(const Args &a, const Tile &T, int ch) {
        return a.tc_cent + (T.c0 / kTcRows + ch) * (int64_t)((a.d + 63) / 64) * kTcBlockBytes;
    }
    struct Epi {
        bool valid;
        float *ls;         // this (query, range)'s list
        int32_t *li;
        float *gm;         // kRankGroupMax: this query's group maxima
        float gacc;        // kRankGroupMax: the running maximum of a 64-centroid group
        int64_t at;        // index of this (query, range)
        int n;             // candidates offered so far
        int bin;           // histogram bin: scores below its lower edge are rejected
        int above;         // kept scores in bins above it (saturated counts)
        float init;        // the starting threshold, raw units
        float edge;        // the threshold in force: max(init, lower edge of bin), raw units
        unsigned char *h;  // this query's bin counts, saturating at 255
        __device__ void begin(const Args &a, const Tile &T, int slot, unsigned char *smem) {
            valid = slot < T.ni;
            const int64_t q = T.q0 + slot;
            at = q * a.nranges + T.c0 / a.range_len;
            n = 0;
            bin = 0;
            above = 0;
            gacc = -__int_as_float(0x7f800000);
            h = kMode == kRankStream ? smem + (size_t)slot * kRankBinStride : nullptr;
            if constexpr (kMode == kRankStream) {
                uint32_t *hw = reinterpret_cast<uint32_t *>(h);
#pragma unroll
                for (int i = 0; i < kRankBins / 4; ++i) hw[i] = 0u;
            }
            init = (valid && a.init_edge) ? a.init_edge[q] * 65536.f : rank_edge_raw(0);
            edge = init;
            ls = valid ? a.list_s + at * a.cap : nullptr;
            li = (valid && a.list_i) ? a.list_i + at * a.cap : nullptr;
            gm = (valid && kMode == kRankGroupMax) ? a.gmax + q * a.gld + T.c0 / a.group : nullptr;
        }
        // v holds the chunk's raw accumulator values: scores x 2^16, for
        // centroids T.c0 + col0 + j, j < ncol (warp-uniform)
        __device__ void chunk(const Args &a, const Tile &T, int64_t col0, const float (&v)[32], int ncol) {
            constexpr float kS = 1.f / 65536.f;
            if (ncol <= 0) return;   // a group past the range's end (warp-uniform)
            if constexpr (kMode == kRankDense) {   // the range's scores in order; ids implicit
                if (!valid) return;
                float *dst = ls + col0;
                if (ncol == 32) {   // cap and the range start are multiples of 32
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        reinterpret_cast<float4 *>(dst)[j] = make_float4(
                            v[4 * j] * kS, v[4 * j + 1] * kS, v[4 * j + 2] * kS, v[4 * j + 3] * kS);
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < ncol) dst[j] = v[j] * kS;
                }
                n += ncol;
                return;
            }
            if constexpr (kMode == kRankStreamInit) {
                // a starting threshold from the first pass: it already keeps
                // only a little over nprobe scores, so no running histogram.
                // The mask comes straight from the compares (some lane of a
                // warp nearly always has a candidate in a group, so a maximum
                // test first would not let the warp skip it)
                unsigned m = 0;
                if (valid) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) m |= v[j] >= edge ? (1u << j) : 0u;
                    if (ncol < 32) m &= (1u << ncol) - 1u;
                }
                const int32_t id0 = (int32_t)(T.c0 + col0);
                while (m) {
                    const int j = __ffs(m) - 1;
                    m &= m - 1u;
                    if (n < a.cap) {
                        ls[n] = pick32(v, j) * kS;
                        li[n] = id0 + j;
                    }
                    ++n;   // counted past cap: an overflow is seen, not lost
                }
                return;
            }
            float mx = v[0];
            if (ncol == 32) {
                mx = max_of_32(v);
            } else {
#pragma unroll
                for (int j = 1; j < 32; ++j) mx = j < ncol ? fmaxf(mx, v[j]) : mx;
            }
            if constexpr (kMode == kRankGroupMax) {
                if (!valid) return;
                if (a.group == 32) {
                    gm[col0 / 32] = mx * kS;
                } else {   // 64: two consecutive 32-column groups (col0 = 0, 32, 64, 96 in turn)
                    gacc = (col0 & 32) ? fmaxf(gacc, mx) : mx;
                    if ((col0 & 32) || ncol < 32 || col0 + 32 >= T.nb) gm[col0 / 64] = gacc * kS;
                }
                return;
            }
            const bool any = valid && mx >= edge;
            if (!__any_sync(0xffffffffu, any)) return;   // the common case: the group is rejected
            unsigned m = 0;
            if (any) {
#pragma unroll
                for (int j = 0; j < 32; ++j) m |= v[j] >= edge ? (1u << j) : 0u;
                if (ncol < 32) m &= (1u << ncol) - 1u;
            }
            const int32_t id0 = (int32_t)(T.c0 + col0);
            while (m) {
                const int j = __ffs(m) - 1;
                m &= m - 1u;
                const float x = pick32(v, j);
                if (!(x >= edge)) continue;   // the threshold rose within this group
                if (n < a.cap) {
                    ls[n] = x * kS;
                    li[n] = id0 + j;
                }
                ++n;   // counted past cap: an overflow is seen, not lost
                const int b = rank_bin(x);   // >= bin, since x reaches the bin's edge
                if (h[b] < 255) {            // a saturated bin stops counting (conservative)
                    ++h[b];
                    if (b > bin && ++above >= a.nprobe) {
                        // nprobe kept scores lie above the threshold bin: raise it
                        while (above >= a.nprobe && bin < kRankBins - 1) {
                            ++bin;
                            above -= h[bin];
                        }
                        edge = fmaxf(init, rank_edge_raw(bin));
                    }
                }
            }
        }
        __device__ void prefetch(const Args &, const Tile &, int) {}
        __device__ void start(const Args &, const Tile &, int) {}
        __device__ void end(const Args &a, const Tile &) {
            if (!valid || kMode == kRankGroupMax || !a.list_n) return;
            a.list_n[at] = n;
            a.list_edge[at] = edge * (1.f / 65536.f);   // exact (-inf stays -inf)
        }
    };
};
// the first pass on the bulk pipeline: one fp16 product per score (hi halves
// of A and B), whose error the threshold allows for; two sub-tiles of 128
// queries share every B stage
struct RankScreenMode : RankModeT<kRankGroupMax, 2> {
    static constexpr int kProducts = 1;
};
// d <= 128: chunks of 192 centroids (MMA N = 192), two sub-tiles' A and two
// 192-column accumulators filling tensor memory; a third fewer MMA
// instructions per score than 128-centroid chunks
struct RankScreen192Mode : RankScreenMode {
    static constexpr int kNB = 192;
};
static_assert(kTcRows == RankModeT<kRankStream>::kN, "");

template <int kMode>
__global__ void __launch_bounds__(tcp::kThreads, 1) k_rank_tc(RankArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcp::run_pipeline<RankModeT<kMode>>(a, smem_raw);
}

int rank_bulk_stages(int d) {
    return tcb::stages_for((int)ceil_div(d, 64), kRankEpiBytes, 232448 - 128);
}

// every pair's screened score (one fp16 product of the hi halves) in a dense
// row per query: a diagnostic of the first pass's arithmetic
struct RankScreenDenseMode : RankModeT<kRankDense> {
    static constexpr int kProducts = 1;
};

__global__ void __launch_bounds__(tcb::kThreads, 1) k_rank_screen_dense(RankArgs a, int stages) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RankScreenDenseMode>(a, smem_raw, stages);
}

template <int kMode, int kSub = 1>
__global__ void __launch_bounds__(tcb::kThreads, 1) k_rank_bulk(RankArgs a, int stages) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RankModeT<kMode, kSub>>(a, smem_raw, stages);
}

// the streaming pass from a starting threshold with two sub-tiles: A of both
// (hi and lo) must leave two accumulators of tensor memory, d <= 128
int rank_pair_stages(int d) {
    const int nkb = (int)ceil_div(d, 64);
    return tcb::sub_fits(nkb, 3, 2) ? tcb::stages_for(nkb, 0, 232448 - 128) : 0;
}

// whether the screen takes 192-centroid chunks (d <= 128), and its B stage bytes
static bool screen_wide(int d) { return ceil_div(d, 64) <= 2; }
static uint32_t screen_stage_bytes(int d) {
    return screen_wide(d) ? tcb::kStageBytesHi / tcb::kN * 192 : tcb::kStageBytesHi;
}

int rank_screen_stages(int d) {
    const int nkb = (int)ceil_div(d, 64);
    return tcb::sub_fits(nkb, 1, 2) ? tcb::stages_for(nkb, 0, 232448 - 128, screen_stage_bytes(d)) : 0;
}

__global__ void __launch_bounds__(tcb::kThreads, 1) k_rank_screen(RankArgs a, int stages) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RankScreenMode>(a, smem_raw, stages);
}

__global__ void __launch_bounds__(tcb::kThreads, 1) k_rank_screen192(RankArgs a, int stages) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RankScreen192Mode>(a, smem_raw, stages);
}

constexpr int kSelectWarps = 4;  // warps (queries) per block of the final selection
constexpr int kSelectMaxR = 8;   // lane order statistics used for the lower bracket

// warp-wide reductions in one instruction (redux.sync), not a chain of shuffles
__device__ __forceinline__ int warp_sum(int x) { return __reduce_add_sync(0xffffffffu, x); }

template <int KPL>
__device__ __forceinline__ int count_ge(const uint32_t (&key)[KPL], uint32_t t) {
    int c = 0;
#pragma unroll
    for (int j = 0; j < KPL; ++j) c += key[j] >= t;
    return warp_sum(c);
}

// A bracket L <= T* <= U of the want-th largest of the warp's keys (keys of
// padding are 0, below every score): U = the largest key, L = the smallest over
// lanes of each lane's ceil(want / 32)-th largest key, so at least want keys
// are >= L.  L = 0 when that rank is past kSelectMaxR.
template <int KPL>
__device__ __forceinline__ void warp_bracket(const uint32_t (&key)[KPL], int want, uint32_t &L,
                                             uint32_t &U) {
    const int r = (want + 31) / 32;
    uint32_t m[kSelectMaxR] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
    if (r <= 2) {
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            m[1] = max(m[1], min(m[0], key[j]));
            m[0] = max(m[0], key[j]);
        }
    } else if (r <= 4) {
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            uint32_t x = key[j];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t hi = max(m[i], x);
                x = min(m[i], x);
                m[i] = hi;
            }
        }
    } else if (r <= kSelectMaxR) {
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            uint32_t x = key[j];
#pragma unroll
            for (int i = 0; i < kSelectMaxR; ++i) {
                const uint32_t hi = max(m[i], x);
                x = min(m[i], x);
                m[i] = hi;
            }
        }
    } else {   // no lower bracket, but U is still the largest key
#pragma unroll
        for (int j = 0; j < KPL; ++j) m[0] = max(m[0], key[j]);
    }
    L = 0u;
#pragma unroll
    for (int i = 0; i < kSelectMaxR; ++i) L = r == i + 1 ? m[i] : L;
    U = __reduce_max_sync(0xffffffffu, m[0]);
    L = __reduce_min_sync(0xffffffffu, L);
}

// A threshold T <= T* (T* = the want-th largest of the warp's keys) with C =
// #{keys >= T} >= want, refined bit by bit (the largest T with at least want
// keys >= T) until C <= cap or T == T*.  The search starts from the common
// high bits of the bracket L, U.
template <int KPL>
__device__ __forceinline__ void warp_threshold(const uint32_t (&key)[KPL], int want, int cap,
                                               uint32_t &T, int &C) {
    uint32_t L, U;
    warp_bracket(key, want, L, U);
    int b;
    if (L == U) {
        b = -1;
        T = L;
    } else {
        b = 31 - __clz(L ^ U);                                // highest bit where they differ
        T = b == 31 ? 0u : (L & ~((2u << b) - 1u));           // their common high bits
    }
    C = count_ge(key, T);
    for (; b >= 0 && C > cap; --b) {
        const uint32_t t = T | (1u << b);
        const int c = count_ge(key, t);
        if (c >= want) {
            T = t;
            C = c;
        }
    }
}

// Bitonic sort of the warp's R * 32 entries (entry i = r * 32 + lane in
// register r), first-ranked first by (score desc, id asc).  Partners within a
// register are exchanged by shuffles, partners across registers in place.
// Entries are distinct except identical padding, so both sides of a pair
// take the same decision.
template <int R>
__device__ __forceinline__ void warp_sort_regs(float (&s)[R], int (&c)[R]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int k = 2; k <= 32 * R; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
            if (j >= 32) {
                const int jr = j >> 5;
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    if (r & jr) continue;
                    const int r2 = r | jr;
                    const bool up = ((r * 32) & k) == 0;   // this block sorts first-ranked first
                    // the lower entry keeps the better one when up, else the worse
                    const bool swap = up ? ranks_before(s[r2], c[r2], s[r], c[r])
                                         : ranks_before(s[r], c[r], s[r2], c[r2]);
                    if (swap) {
                        const float ts = s[r];
                        const int tc = c[r];
                        s[r] = s[r2];
                        c[r] = c[r2];
                        s[r2] = ts;
                        c[r2] = tc;
                    }
                }
            } else {
                const bool lower = (lane & j) == 0;
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const float ps = __shfl_xor_sync(0xffffffffu, s[r], j);
                    const int pc = __shfl_xor_sync(0xffffffffu, c[r], j);
                    const bool up = (((r * 32) + lane) & k) == 0;
                    const bool take = (lower == up) ? ranks_before(ps, pc, s[r], c[r])
                                                    : ranks_before(s[r], c[r], ps, pc);
                    if (take) {
                        s[r] = ps;
                        c[r] = pc;
                    }
                }
            }
        }
    }
}

// Sort bs/bc[0 .. want-1] in place (R * 32 >= want entries; the rest become
// padding (-inf, INT32_MAX))
template <int R>
__device__ __forceinline__ void sort_buffer(float *bs, int *bc, int want) {
    const int lane = threadIdx.x & 31;
    float s[R];
    int c[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int i = r * 32 + lane;
        s[r] = i < want ? bs[i] : -__int_as_float(0x7f800000);
        c[r] = i < want ? bc[i] : INT32_MAX;
    }
    __syncwarp();
    warp_sort_regs<R>(s, c);
#pragma unroll
    for (int r = 0; r < R; ++r) {
        bs[r * 32 + lane] = s[r];
        bc[r * 32 + lane] = c[r];
    }
    __syncwarp();
}

// The want best of the warp's cnt entries (entry c = key[c / 32] of lane
// c % 32, its id from id_of(c)) into bs/bc[0 .. want-1], in entry order,
// given T and C from warp_threshold(key, want, want, ..); id_of(j, c) is the
// id of entry c = j * 32 + lane.  C == want: every
// key >= T.  Otherwise T == T* and the keys > T* plus the first keys equal to
// it in entry order are taken, which are the lowest ids when entry order is id
// order among equal scores.
template <int KPL, class IdOf>
__device__ __forceinline__ void warp_gather_exact(const uint32_t (&key)[KPL], int cnt, int want,
                                                  uint32_t T, int C, IdOf id_of, float *bs,
                                                  int *bc) {
    const int lane = threadIdx.x & 31;
    const unsigned below = (1u << lane) - 1u;
    const bool ties = C > want;
    int ties_wanted = 0;
    if (ties) {
        int gt = 0;
#pragma unroll
        for (int j = 0; j < KPL; ++j) gt += key[j] > T && j * 32 + lane < cnt;
        ties_wanted = want - warp_sum(gt);   // >= 1
    }
    int pos = 0, ties_seen = 0;
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        const bool in = c < cnt;
        bool sel;
        if (ties) {
            const bool tie = key[j] == T && in;
            const unsigned tb = __ballot_sync(0xffffffffu, tie);
            sel = (key[j] > T && in) || (tie && ties_seen + __popc(tb & below) < ties_wanted);
            ties_seen += __popc(tb);
        } else {
            sel = key[j] >= T && in;
        }
        const unsigned sb = __ballot_sync(0xffffffffu, sel);
        if (sel) {
            const int p = pos + __popc(sb & below);
            if (p < want) {   // exactly want are selected; the bound guards the buffer
                bs[p] = key_score(key[j]);
                bc[p] = id_of(j, c);
            }
        }
        pos += __popc(sb);
    }
    __syncwarp();
}

// the want best of n candidates (keys ck, ids ci in shared memory, id order;
// n <= 32 * KPL, want <= n) into bs/bc, in id order
template <int KPL>
__device__ __forceinline__ void select_candidates(const uint32_t *ck, const int *ci, int n, int want,
                                                  float *bs, int *bc) {
    const int lane = threadIdx.x & 31;
    uint32_t key[KPL];
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        key[j] = c < n ? ck[c] : 0u;
    }
    uint32_t T;
    int C;
    warp_threshold(key, want, want, T, C);
    warp_gather_exact(key, n, want, T, C, [&](int, int c) { return ci[c]; }, bs, bc);
}

// The want best of the warp's cnt entries (KPL keys per lane, entry c =
// key[c / 32] of lane c % 32, its id id_of(c)) into bs/bc in entry order, in
// two steps: a first threshold refined until at most 32 * K2 keys reach it
// (K2 about 2 want / 32), those keys compacted in entry order into ck/ci, and
// the exact selection over K2 keys per lane.  A first threshold still
// reached by more than 32 * K2 keys is the want-th largest key itself, tied:
// the exact gather over all keys takes it from there.
template <int K2, int KPL, class IdOf>
__device__ __forceinline__ void select_two_step(const uint32_t (&key)[KPL], int cnt, int want,
                                                IdOf id_of, uint32_t *ck, int *ci, float *bs,
                                                int *bc) {
    uint32_t T;
    int C;
    warp_threshold(key, want, 32 * K2, T, C);
    if (C > 32 * K2) {
        warp_gather_exact(key, cnt, want, T, C, id_of, bs, bc);
        return;
    }
    const int lane = threadIdx.x & 31;
    const unsigned below = (1u << lane) - 1u;
    int pos = 0;
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        const bool sel = key[j] >= T && c < cnt;
        const unsigned sb = __ballot_sync(0xffffffffu, sel);
        if (sel) {
            const int p = pos + __popc(sb & below);
            ck[p] = key[j];
            ci[p] = id_of(j, c);
        }
        pos += __popc(sb);
    }
    __syncwarp();
    uint32_t k2[K2];
#pragma unroll
    for (int j = 0; j < K2; ++j) {
        const int c = j * 32 + lane;
        k2[j] = c < pos ? ck[c] : 0u;
    }
    warp_threshold(k2, want, want, T, C);
    warp_gather_exact(k2, pos, want, T, C, [&](int, int c) { return ci[c]; }, bs, bc);
}

constexpr int kDenseK2Max = 16;   // second-step keys per lane of the dense selection

// One warp per query of a dense single-range ranking (every score of the
// query in its list, ids = positions): the keys straight from the list into
// registers (KPL per lane), the nprobe best (two steps when KPL > 16), sorted.
template <int KPL, int R>
__global__ void __launch_bounds__(kSelectWarps * 32, (KPL >= 64 || R >= 8) ? 4 : 8) k_rank_dense_final(
    const float *__restrict__ list_s, const int *__restrict__ list_n, int64_t nq, int cap,
    int nprobe, int32_t *__restrict__ order, float *__restrict__ cscores) {
    extern __shared__ __align__(16) unsigned char sel_smem[];
    constexpr int kK2 = R <= 2 ? 4 : R == 4 ? 8 : kDenseK2Max;   // about twice nprobe / 32
    constexpr int kSort = 32 * R;
    constexpr int kS2 = KPL > kDenseK2Max ? 32 * kK2 : 0;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *bs = reinterpret_cast<float *>(sel_smem) + (size_t)warp * 2 * (kSort + kS2);
    int *bc = reinterpret_cast<int *>(bs + kSort);
    uint32_t *ck = reinterpret_cast<uint32_t *>(bc + kSort);
    int *ci = reinterpret_cast<int *>(ck + kS2);
    const int64_t q = (int64_t)blockIdx.x * kSelectWarps + warp;
    if (q >= nq) return;
    const float *row = list_s + q * cap;
    const int cnt = list_n[q];
    const int want = nprobe < cnt ? nprobe : cnt;
    uint32_t key[KPL];
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        key[j] = c < cnt ? order_key(row[c]) : 0u;   // padding ranks below every score
    }
    auto id_of = [](int, int c) { return c; };
    if constexpr (KPL > kDenseK2Max) {
        select_two_step<kK2>(key, cnt, want, id_of, ck, ci, bs, bc);
    } else {
        uint32_t T;
        int C;
        warp_threshold(key, want, want, T, C);
        warp_gather_exact(key, cnt, want, T, C, id_of, bs, bc);
    }
    sort_buffer<R>(bs, bc, want);
    for (int p = lane; p < nprobe; p += 32) {
        order[q * nprobe + p] = p < want ? bc[p] : INT32_MAX;
        if (cscores) cscores[q * nprobe + p] = p < want ? bs[p] : -__int_as_float(0x7f800000);
    }
}

static size_t dense_smem(int kpl, int R) {
    const int k2 = R <= 2 ? 4 : R == 4 ? 8 : kDenseK2Max;
    return (size_t)kSelectWarps * 2 * (32 * (size_t)R + (kpl > kDenseK2Max ? 32 * (size_t)k2 : 0)) * 4;
}

// One warp per query: the candidates of its ranges that reach their final
// thresholds, gathered in order (id order) into ccap slots, then the nprobe
// best sorted into order/cscores.  Dense lists (list_i null) hold every score
// of their range, the id being the range start plus the position.  A list past cap, more than ccap
// candidates, or fewer than nprobe (NaN scores): the query is appended to
// ovf_list (count in *ovf_n, zeroed before the launch) for the exact FP32
// ranking.  nprobe <= 32 * R.
template <int R, int KMAX>   // KMAX: keys per lane of the largest candidate set (ccap / 32)
__global__ void __launch_bounds__(kSelectWarps * 32, KMAX <= 16 ? 8 : 4) k_rank_final(
    const float *__restrict__ list_s, const int32_t *__restrict__ list_i,
    const int *__restrict__ list_n, const float *__restrict__ list_edge, int64_t nq, int nranges,
    int64_t range_len, int cap, int nprobe, int ccap, int32_t *__restrict__ order,
    float *__restrict__ cscores, int *__restrict__ ovf_list, int *__restrict__ ovf_n) {
    extern __shared__ __align__(16) unsigned char sel_smem[];
    constexpr int kSort = 32 * R;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char *wbase = sel_smem + (size_t)warp * ((size_t)ccap + kSort) * 8;
    uint32_t *ck = reinterpret_cast<uint32_t *>(wbase);                 // candidate keys
    int *ci = reinterpret_cast<int *>(wbase + (size_t)ccap * 4);        // candidate ids
    float *bs = reinterpret_cast<float *>(wbase + (size_t)ccap * 8);    // sort buffer
    int *bc = reinterpret_cast<int *>(bs + kSort);
    const int64_t q = (int64_t)blockIdx.x * kSelectWarps + warp;
    if (q >= nq) return;
    const unsigned below = (1u << lane) - 1u;
    int n = 0;
    bool over = false;
    for (int r = 0; r < nranges && !over; ++r) {
        const int64_t at = q * nranges + r;
        const int cnt = list_n[at];
        if (cnt > cap) {
            over = true;
            break;
        }
        const float e = list_edge[at];
        const float *s = list_s + at * cap;
        const int32_t *id = list_i ? list_i + at * cap : nullptr;   // null: dense, id = position
        const int32_t id0 = (int32_t)(r * range_len);
        for (int i0 = 0; i0 < cnt; i0 += 32) {
            const int i = i0 + lane;
            const float x = i < cnt ? s[i] : 0.f;
            const bool keep = i < cnt && x >= e;
            const unsigned bal = __ballot_sync(0xffffffffu, keep);
            const int p = n + __popc(bal & below);
            if (keep && p < ccap) {
                ck[p] = order_key(x);
                ci[p] = id ? id[i] : id0 + i;
            }
            n += __popc(bal);
        }
        over = n > ccap;
    }
    if (over || n < nprobe) {
        if (lane == 0) ovf_list[atomicAdd(ovf_n, 1)] = (int)q;
        return;
    }
    __syncwarp();
    // keys per lane sized to the candidates (warp-uniform n <= ccap <= 32 KMAX)
    if (n <= 128 || KMAX <= 4)
        select_candidates<4>(ck, ci, n, nprobe, bs, bc);
    else if (n <= 512 || KMAX <= 16)
        select_candidates<(KMAX < 16 ? KMAX : 16)>(ck, ci, n, nprobe, bs, bc);
    else if (n <= 1024 || KMAX <= 32)
        select_candidates<(KMAX < 32 ? KMAX : 32)>(ck, ci, n, nprobe, bs, bc);
    else
        select_candidates<KMAX>(ck, ci, n, nprobe, bs, bc);
    sort_buffer<R>(bs, bc, nprobe);
    for (int p = lane; p < nprobe; p += 32) {
        order[q * nprobe + p] = bc[p];
        if (cscores) cscores[q * nprobe + p] = bs[p];
    }
}

// The largest centroid norm (one float, zeroed before the launch; norms are
// non-negative, so their bit patterns order like the floats)
__global__ void k_cnorm_max(const float *__restrict__ C, int64_t nlist, int d,
                            unsigned *__restrict__ out) {
    const int lane = threadIdx.x & 31;
    float best = 0.f;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; c < nlist; c += warps) {
        float ss = 0.f;
        for (int t = lane; t < d; t += 32) ss = fmaf(C[c * d + t], C[c * d + t], ss);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        best = fmaxf(best, sqrtf(ss));
    }
    if (lane == 0) atomicMax(out, __float_as_uint(best));
}

// One warp per query: T = a key reached by at least nprobe of its ng group
// maxima (warp_threshold; each maximum is a different centroid's score), so
// at least nprobe centroids score >= T in the first pass.  The second pass
// keeps every score >= T - margin, margin = the first pass's error bound plus
// the second's (slack = 0 when both passes compute identical scores):
//   screen (one fp16 product of the hi halves, fp32 sums, as in the screening
//   scan): (2^-10 + 2^-12 + d 2^-22) |q| |c| + 2^-26 sqrt(d) (|q| + |c|);
//   three products: (2^-20 + d 2^-22) |q| |c| + 2^-26 sqrt(d) (|q| + |c|)
//   (the dropped lo*lo term and the rounding of the lo halves, 3 2^-22 of each
//   |q_i c_i|, and the fp32 sums of 3d products);
// |c| = the largest centroid norm.  Every centroid among the nprobe best of
// the second pass then scores >= T - margin: the nprobe centroids with a
// first-pass score >= T score at least T - margin there.  Writes the
// starting threshold (score units) of each query.
template <int KPL>
__global__ void __launch_bounds__(kSelectWarps * 32) k_rank_threshold(
    const float *__restrict__ gmax, int64_t gld, int64_t nq, int ng, int nprobe,
    const float *__restrict__ Q, int d, const unsigned *__restrict__ cmax_bits, int screen,
    float *__restrict__ init_edge) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t q = (int64_t)blockIdx.x * kSelectWarps + warp;
    if (q >= nq) return;
    const float *row = gmax + q * gld;
    uint32_t key[KPL];
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        key[j] = c < ng ? order_key(row[c]) : 0u;
    }
    uint32_t T;
    int C;
    warp_threshold(key, nprobe, nprobe, T, C);
    float ss = 0.f;
    for (int t = lane; t < d; t += 32) ss = fmaf(Q[q * d + t], Q[q * d + t], ss);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    // the norms and the margin rounded upward, so the margin is never short
    const float qn = __fsqrt_ru(ss) * (1.f + 0x1p-20f);
    const float cn = __uint_as_float(*cmax_bits) * (1.f + 0x1p-20f);
    const float rd = __fsqrt_ru((float)d);
    const float three = (0x1p-20f + (float)d * 0x1p-22f) * qn * cn + 0x1p-26f * rd * (qn + cn);
    const float scr = screen ? (0x1p-10f + 0x1p-12f + (float)d * 0x1p-22f) * qn * cn +
                                   0x1p-26f * rd * (qn + cn)
                             : 0.f;
    const float margin = screen ? (scr + three) * (1.f + 0x1p-16f) : 0.f;
    if (lane == 0) init_edge[q] = __fsub_rd(key_score(T), margin);
}

// ---------------------------------------------------------------------------
cudaError_t enqueue_screen_scores(const float *Q, int64_t nq, int64_t nlist, int d,
                                  const unsigned char *tc_cent, float *out, int64_t ld,
                                  int *status, cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    const int nkb = (int)ceil_div(d, 64);
    const int stages = tcb::stages_for(nkb, 0, 232448 - 128, tcb::kStageBytesHi);
    if (stages == 0) return cudaErrorInvalidValue;
    const size_t smem = tcb::smem_bytes(stages, 0, tcb::kStageBytesHi);
    cudaError_t e = cudaFuncSetAttribute(k_rank_screen_dense, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    RankArgs a{};
    a.Q = Q;
    a.nq = nq;
    a.nlist = nlist;
    a.d = d;
    a.status = status;
    a.tc_cent = tc_cent;
    a.nprobe = 1;
    a.nranges = 1;
    a.range_len = round_up(nlist, (int64_t)kTcRows);
    a.cap = (int)ld;
    a.list_s = out;
    const int tiles = (int)ceil_div(nq, tcp::kM);
    k_rank_screen_dense<<<(unsigned)std::min(tiles, num_sms()), tcb::kThreads, smem, st>>>(a, stages);
    return cudaGetLastError();
}

bool rank_tc_supported(int64_t nlist, int nprobe) { return nlist >= 1 && nprobe <= nlist; }

static int pow2_at_least(int64_t x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

// registers per lane of the sort of nprobe entries
static int sort_regs(int nprobe) { return std::max(2, pow2_at_least(nprobe) / 32); }

constexpr int kFinalCapMax = 2048;   // candidates one final-selection warp holds (64 per lane)
constexpr int kMaxGroups = 2048;     // group maxima one threshold warp holds (64 per lane)

// How one ranking call is cut up.
//  kind: nlist <= 2,048: one pass keeping every score (dense lists, ids
//    implicit).  Else, on the bulk pipeline with at least 2 nprobe groups of
//    64 (or 32) centroids and at most 2,048 of them: two passes -- group
//    maxima on the screen, a per-query threshold, and the streaming pass
//    from that threshold.  Else the streaming pass alone.
//  ranges: enough (query tile, range) tiles for about four waves of the
//    persistent contraction; the streaming pass alone takes at most
//    2,048 / 2P ranges (each keeps P plus a bin's width of candidates);
//  cap: list slots per (query, range): the whole range (dense); 2P, at least
//    256 (two passes: the threshold keeps a little over P per query in all);
//    with the running threshold alone, a random order offers about
//    P (1 + ln(len / P)) scores (the expected number of times a new score
//    enters the running best P, standard deviation near sqrt(P ln(len / P))),
//    and the cap is 1.25 times that plus 64, at most 8,192;
//  chunk: queries per pass, so that their scratch fits kRankScratchBytes.
struct RankPlan {
    int mode;        // the final pass: kRankDense or kRankStream
    int group;       // centroids per group of the first pass; 0 = no first pass
    bool screen;     // the first pass screens (bulk pipeline)
    int nranges;
    int64_t range_len;
    int cap;
    int ng;          // groups of the first pass
    int64_t gld;
    int ccap;        // final-selection slots
    int64_t chunk;
    int64_t per_query() const {
        const int64_t entry = mode == kRankDense ? 4 : 8;
        return (int64_t)nranges * ((int64_t)cap * entry + 8) + 4 + (group ? gld * 4 + 4 : 0);
    }
};
constexpr int64_t kRankFixedBytes = 256;   // the overflow count and the largest centroid norm

static RankPlan rank_plan(int64_t nq, int64_t nlist, int nprobe, int d, bool bulk) {
    RankPlan L{};
    const int P = pow2_at_least(nprobe);
    L.group = 0;
    if (nlist <= kFinalCapMax) {
        L.mode = kRankDense;
    } else {
        L.mode = kRankStream;
        // a first pass pays off on the screen (a third of the products and
        // half the operand bytes); without the bulk pipeline it would cost a
        // full second contraction
        for (int g : {64, 32}) {
            if (!bulk || rank_screen_stages(d) == 0) break;
            const int64_t ng = ceil_div(nlist, g);
            if (ng >= 2 * (int64_t)nprobe && ng <= kMaxGroups) {
                L.group = g;
                break;
            }
        }
    }
    L.screen = L.group && bulk && rank_screen_stages(d) > 0;
    const int64_t qtiles = std::max<int64_t>(1, ceil_div(nq, tcp::kM));
    const int64_t want = ceil_div(4 * (int64_t)num_sms(), qtiles);
    int64_t most = ceil_div(nlist, RankModeT<kRankStream>::kN);
    if (L.mode == kRankStream && !L.group) most = std::min<int64_t>(most, std::max(1, kFinalCapMax / (2 * P)));
    const int64_t r = std::max<int64_t>(1, std::min(want, most));
    L.range_len = round_up(ceil_div(nlist, r), RankModeT<kRankStream>::kN);
    L.nranges = (int)ceil_div(nlist, L.range_len);
    if (L.mode == kRankDense) {
        L.cap = (int)round_up(L.range_len, 32);
    } else if (L.group) {
        L.cap = std::max(256, 2 * P);
    } else {
        const double offered = P * (1.0 + std::log(std::max(1.0, (double)L.range_len / P)));
        L.cap = (int)std::min<int64_t>(8192, round_up((int64_t)std::ceil(1.25 * offered) + 64, 64));
    }
    L.cap = (int)std::min<int64_t>(L.cap, round_up(L.range_len, 32));
    L.ng = L.group ? (int)ceil_div(nlist, L.group) : 0;
    L.gld = L.group ? round_up(L.ng, 4) : 0;
    L.ccap = (int)std::min<int64_t>(kFinalCapMax, round_up((int64_t)L.nranges * L.cap, 32));
    int64_t c = (kRankScratchBytes - kRankFixedBytes) / L.per_query();
    c = std::max<int64_t>(tcp::kM, c / tcp::kM * tcp::kM);
    L.chunk = std::min(nq, c);
    return L;
}

size_t rank_tc_scratch_bytes(int64_t nq, int64_t nlist, int nprobe, int d) {
    if (nq <= 0) return kRankFixedBytes;
    // the bulk pipeline's plan needs at least the converter's scratch: size for the larger
    const RankPlan a = rank_plan(nq, nlist, nprobe, d, true), b = rank_plan(nq, nlist, nprobe, d, false);
    return (size_t)(std::max(a.chunk * a.per_query(), b.chunk * b.per_query()) + kRankFixedBytes);
}

static size_t tc_smem() { return tcp::Geometry<RankModeT<kRankStream>::kN>::smem_bytes(kRankEpiBytes); }

static size_t final_smem(int ccap, int R) {
    return (size_t)kSelectWarps * ((size_t)ccap + 32 * (size_t)R) * 8;
}

template <int R>
static cudaError_t set_final_attr() {
    cudaError_t e = cudaSuccess;
    for (auto f : {k_rank_final<R, 4>, k_rank_final<R, 16>, k_rank_final<R, 32>, k_rank_final<R, 64>})
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)final_smem(kFinalCapMax, R));
    return e;
}

cudaError_t prepare_rank_tc(int nprobe, int d) {
    cudaError_t e = cudaSuccess;
    for (auto f : {k_rank_tc<kRankGroupMax>, k_rank_tc<kRankStream>, k_rank_tc<kRankDense>})
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc_smem());
    const int bulk = rank_bulk_stages(d);
    for (auto f : {k_rank_bulk<kRankGroupMax>, k_rank_bulk<kRankStream>, k_rank_bulk<kRankDense>,
                   k_rank_bulk<kRankStreamInit>})
        if (e == cudaSuccess && bulk)
            e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tcb::smem_bytes(bulk, kRankEpiBytes));
    const int pair = rank_pair_stages(d);
    if (e == cudaSuccess && pair)
        e = cudaFuncSetAttribute(k_rank_bulk<kRankStreamInit, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)tcb::smem_bytes(pair, 0));
    const int scr = rank_screen_stages(d);
    if (e == cudaSuccess && scr)
        e = cudaFuncSetAttribute(screen_wide(d) ? k_rank_screen192 : k_rank_screen,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)tcb::smem_bytes(scr, 0, screen_stage_bytes(d)));
    if (e == cudaSuccess) e = set_final_attr<2>();
    if (e == cudaSuccess) e = set_final_attr<4>();
    if (e == cudaSuccess) e = set_final_attr<8>();
    if (e == cudaSuccess) e = set_final_attr<16>();
    // the exact fallback for overflowing lists
    if (e == cudaSuccess) e = prepare_rank(nprobe);
    return e;
}

static void launch_final(const RankArgs &a, const RankPlan &L, int64_t n, int32_t *order,
                         float *cscores, int *ovf, int *ovf_n, cudaStream_t st) {
    const unsigned blocks = (unsigned)ceil_div(n, kSelectWarps);
    if (L.mode == kRankDense && L.nranges == 1) {   // every score of a query in one list
        const int kpl = std::max(4, pow2_at_least(ceil_div(L.cap, 32)));
#define SIEVE_DENSE(KK, RR)                                                                      \
    k_rank_dense_final<KK, RR><<<blocks, kSelectWarps * 32, dense_smem(KK, RR), st>>>(              \
        a.list_s, a.list_n, n, a.cap, a.nprobe, order, cscores)
#define SIEVE_DENSE_R(KK)                   \
    switch (sort_regs(a.nprobe)) {          \
        case 2: SIEVE_DENSE(KK, 2); break;  \
        case 4: SIEVE_DENSE(KK, 4); break;  \
        case 8: SIEVE_DENSE(KK, 8); break;  \
        default: SIEVE_DENSE(KK, 16); break; \
    }
        switch (kpl) {
            case 4: SIEVE_DENSE_R(4); break;
            case 8: SIEVE_DENSE_R(8); break;
            case 16: SIEVE_DENSE_R(16); break;
            case 32: SIEVE_DENSE_R(32); break;
            default: SIEVE_DENSE_R(64); break;
        }
#undef SIEVE_DENSE_R
#undef SIEVE_DENSE
        return;
    }
    const int kmax = L.ccap <= 128 ? 4 : L.ccap <= 512 ? 16 : L.ccap <= 1024 ? 32 : 64;
#define SIEVE_FINAL(RR, KK)                                                                      \
    k_rank_final<RR, KK><<<blocks, kSelectWarps * 32, final_smem(L.ccap, RR), st>>>(                \
        a.list_s, a.list_i, a.list_n, a.list_edge, n, a.nranges, a.range_len, a.cap, a.nprobe,    \
        L.ccap, order, cscores, ovf, ovf_n)
#define SIEVE_FINAL_R(RR)                   \
    switch (kmax) {                         \
        case 4: SIEVE_FINAL(RR, 4); break;   \
        case 16: SIEVE_FINAL(RR, 16); break; \
        case 32: SIEVE_FINAL(RR, 32); break; \
        default: SIEVE_FINAL(RR, 64); break; \
    }
    switch (sort_regs(a.nprobe)) {
        case 2: SIEVE_FINAL_R(2); break;
        case 4: SIEVE_FINAL_R(4); break;
        case 8: SIEVE_FINAL_R(8); break;
        default: SIEVE_FINAL_R(16); break;
    }
#undef SIEVE_FINAL_R
#undef SIEVE_FINAL
}

static void launch_threshold(const RankPlan &L, const float *gmax, int64_t n, int nprobe,
                             const float *Q, int d, const unsigned *cmax, float *init_edge,
                             cudaStream_t st) {
    const unsigned blocks = (unsigned)ceil_div(n, kSelectWarps);
    const int kpl = std::max(1, pow2_at_least(ceil_div(L.ng, 32)));
#define SIEVE_THR(K)                                                                             \
    k_rank_threshold<K><<<blocks, kSelectWarps * 32, 0, st>>>(gmax, L.gld, n, L.ng, nprobe, Q, d, \
                                                              cmax, L.screen ? 1 : 0, init_edge)
    switch (kpl) {
        case 1: SIEVE_THR(1); break;
        case 2: SIEVE_THR(2); break;
        case 4: SIEVE_THR(4); break;
        case 8: SIEVE_THR(8); break;
        case 16: SIEVE_THR(16); break;
        case 32: SIEVE_THR(32); break;
        default: SIEVE_THR(64); break;
    }
#undef SIEVE_THR
}

// per chunk of queries: [the first pass and the threshold,] the final pass,
// the final selection and the FP32 fallback; once per call the largest
// centroid norm (the screen's bound)
int rank_tc_launches(int64_t nq, int64_t nlist, int nprobe, int d, int64_t plan_nq,
                     bool bulk) {
    if (nq <= 0) return 0;
    const RankPlan L = rank_plan(std::max(nq, plan_nq), nlist, nprobe, d, bulk);
    const int chunks = (int)ceil_div(nq, L.chunk);
    return chunks * (L.group ? 5 : 3) + (L.screen ? 1 : 0);
}

int rank_tc_mma_launches(int64_t nq, int64_t nlist, int nprobe, int d, int64_t plan_nq,
                         bool bulk) {
    if (nq <= 0) return 0;
    const RankPlan L = rank_plan(std::max(nq, plan_nq), nlist, nprobe, d, bulk);
    return (int)ceil_div(nq, L.chunk) * (L.group ? 2 : 1);
}

cudaError_t enqueue_rank_tc(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                            int nprobe, int32_t *order, float *cscores, float *scratch, int *status,
                            cudaStream_t st, const unsigned char *tc_cent, float *mma_ms,
                            int64_t plan_nq) {
    if (nq <= 0) return cudaSuccess;
    // the layout of the scratch follows the batch it was sized for; a part of
    // that batch uses the same layout, so it never needs more
    if (plan_nq < nq) plan_nq = nq;
    struct Events {   // mma_ms: a pair per contraction launch, destroyed on every return
        std::vector<cudaEvent_t> v;
        ~Events() {
            for (cudaEvent_t e : v) cudaEventDestroy(e);
        }
    } ev_hold;
    std::vector<cudaEvent_t> &evs = ev_hold.v;
    const int bulk_stages = tc_cent ? rank_bulk_stages(d) : 0;
    const RankPlan L = rank_plan(plan_nq, nlist, nprobe, d, bulk_stages > 0);
    const int screen_stages = L.screen ? rank_screen_stages(d) : 0;
    const int pair_stages = bulk_stages && L.group ? rank_pair_stages(d) : 0;
    // the chunk's scratch: lists (scores, ids), counts, final thresholds,
    // overflow list, group maxima, starting thresholds; then the fixed part
    const int64_t slots = L.chunk * L.nranges;
    float *list_s = scratch;
    int32_t *list_i = L.mode == kRankDense ? nullptr : reinterpret_cast<int32_t *>(list_s + slots * L.cap);
    int *list_n = reinterpret_cast<int *>(list_s + slots * L.cap * (L.mode == kRankDense ? 1 : 2));
    float *list_edge = reinterpret_cast<float *>(list_n + slots);
    int *ovf = reinterpret_cast<int *>(list_edge + slots);
    float *gmax = reinterpret_cast<float *>(ovf + L.chunk);
    float *init_edge = gmax + (L.group ? L.chunk * L.gld : 0);
    unsigned char *fixed = reinterpret_cast<unsigned char *>(scratch) + L.chunk * L.per_query();
    int *ovf_n = reinterpret_cast<int *>(fixed);
    unsigned *cmax = reinterpret_cast<unsigned *>(fixed + 4);
    auto contract = [&](int mode, const RankArgs &a, int64_t n, bool scr) {
        if (mma_ms) {
            evs.resize(evs.size() + 2);
            cudaEventCreate(&evs[evs.size() - 2]);
            cudaEventCreate(&evs.back());
            cudaEventRecord(evs[evs.size() - 2], st);
        }
        // tiles of 128 queries, or of two sub-tiles of 128 (the screen, and the
        // streaming pass from a starting threshold where A fits twice)
        const bool two = scr || (mode == kRankStreamInit && pair_stages);
        const int tiles = (int)(ceil_div(n, (two ? 2 : 1) * tcp::kM) * L.nranges);
        const unsigned grid = (unsigned)std::min(tiles, num_sms());
        const size_t bsm = tcb::smem_bytes(bulk_stages, kRankEpiBytes);
        if (scr && screen_wide(d))
            k_rank_screen192<<<grid, tcb::kThreads, tcb::smem_bytes(screen_stages, 0, screen_stage_bytes(d)),
                               st>>>(a, screen_stages);
        else if (scr)
            k_rank_screen<<<grid, tcb::kThreads, tcb::smem_bytes(screen_stages, 0, tcb::kStageBytesHi),
                            st>>>(a, screen_stages);
        else if (mode == kRankStreamInit && pair_stages)
            k_rank_bulk<kRankStreamInit, 2><<<grid, tcb::kThreads, tcb::smem_bytes(pair_stages, 0), st>>>(
                a, pair_stages);
        else if (mode == kRankStreamInit)
            k_rank_bulk<kRankStreamInit><<<grid, tcb::kThreads, bsm, st>>>(a, bulk_stages);
        else if (bulk_stages && mode == kRankGroupMax)
            k_rank_bulk<kRankGroupMax><<<grid, tcb::kThreads, bsm, st>>>(a, bulk_stages);
        else if (bulk_stages && mode == kRankStream)
            k_rank_bulk<kRankStream><<<grid, tcb::kThreads, bsm, st>>>(a, bulk_stages);
        else if (bulk_stages)
            k_rank_bulk<kRankDense><<<grid, tcb::kThreads, bsm, st>>>(a, bulk_stages);
        else if (mode == kRankGroupMax)
            k_rank_tc<kRankGroupMax><<<grid, tcp::kThreads, tc_smem(), st>>>(a);
        else if (mode == kRankStream)
            k_rank_tc<kRankStream><<<grid, tcp::kThreads, tc_smem(), st>>>(a);
        else
            k_rank_tc<kRankDense><<<grid, tcp::kThreads, tc_smem(), st>>>(a);
        if (mma_ms) cudaEventRecord(evs.back(), st);
    };
    if (L.screen) {
        cudaError_t e = cudaMemsetAsync(cmax, 0, sizeof(unsigned), st);
        if (e != cudaSuccess) return e;
        const unsigned blocks = (unsigned)std::min<int64_t>(ceil_div(nlist, 8), 4 * (int64_t)num_sms());
        k_cnorm_max<<<blocks, 256, 0, st>>>(C, nlist, d, cmax);
    }
    for (int64_t q0 = 0; q0 < nq; q0 += L.chunk) {
        const int64_t n = nq - q0 < L.chunk ? nq - q0 : L.chunk;
        RankArgs a{Q + q0 * d, n, C, nlist, d, status, tc_cent, nprobe, L.nranges,
                   L.range_len, L.cap, list_s, list_i, list_n, list_edge, nullptr, gmax, L.gld,
                   L.group};
        if (L.group) {   // the first pass: group maxima, then each query's starting threshold
            contract(kRankGroupMax, a, n, L.screen);
            launch_threshold(L, gmax, n, nprobe, Q + q0 * d, d, cmax, init_edge, st);
            a.init_edge = init_edge;
        }
        contract(L.group ? kRankStreamInit : L.mode, a, n, false);
        cudaError_t e = cudaMemsetAsync(ovf_n, 0, sizeof(int), st);
        if (e != cudaSuccess) return e;
        int32_t *o = order + q0 * nprobe;
        float *cs = cscores ? cscores + q0 * nprobe : nullptr;
        launch_final(a, L, n, o, cs, ovf, ovf_n, st);
        // the queries whose lists overflowed: the FP32 ranking, exact
        e = enqueue_rank(Q + q0 * d, n, C, nlist, d, nprobe, o, cs, st, ovf, ovf_n);
        if (e != cudaSuccess) return e;
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (mma_ms) {
        cudaError_t e = cudaStreamSynchronize(st);
        for (size_t i = 0; i + 1 < evs.size(); i += 2) {
            float t = 0.f;
            if (e == cudaSuccess) e = cudaEventElapsedTime(&t, evs[i], evs[i + 1]);
            *mma_ms += t;
        }
        return e;
    }
    return cudaSuccess;
}

}  // namespace sieve
