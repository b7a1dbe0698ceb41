// rank_tc.cu -- centroid ranking on the tcgen05 tensor cores (Sec. 2.3,
// Sec. 4.1: P_i = the nprobe centroids with the largest inner product with
// q_i, best first, equal scores by lower centroid id), for any nlist.
//
// Per chunk of queries:
//   k_rank_bulk / k_rank_tc  the tensor-core contraction (tc_bulk.cuh with the
//              centroids' tensor-core layout, else the converter pipeline of
//              tc_pipeline.cuh): a tile is 128 consecutive queries (A rows)
//              against one range of kRankRange centroids (B rows, 128 per
//              chunk); each epilogue thread owns one query's scores and stores
//              them into a score table, or only the maxima of 32-centroid
//              groups, or only the scores that reach the query's threshold
//   k_select   one warp per (query, segment of at most kSelectSeg entries):
//              the segment's best min(nprobe, size) entries, sorted by
//              (score desc, id asc): a threshold refined bit by bit over the
//              keys in registers picks exactly that many, and a bitonic
//              network in registers sorts them.  With nlist <= kSelectSeg one
//              segment gives the order directly.
// More centroids: the nprobe-th largest of the 32-centroid group maxima is a
// threshold that at least nprobe scores reach (k_group_threshold); the scores
// that reach it are compacted per 2,048-centroid range (from the table by
// k_compact_seg, or kept by a second contraction when d <= 128) and one warp
// per query selects and sorts the nprobe best of them (k_compact_final).  A
// query whose candidates overflow their slots is listed and finished exactly:
// by levels of k_select over its table row (the nprobe best of a set lie among
// the nprobe best of each of its parts), or by the FP32 ranking of
// rank_kernel.cu when there is no table.
#include <vector>

#include "tc_bulk.cuh"
#include "tc_pipeline.cuh"

namespace sieve {

constexpr int64_t kRankRange = 2048;   // centroids per tile (a multiple of 128)
constexpr int kSelectSeg = 2048;       // entries per selecting warp (64 per lane)

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


struct RankArgs {
    const float *Q;
    int64_t nq;
    const float *C;
    int64_t nlist;
    int d;
    float *scores;   // [nq][ld] score table
    int64_t ld;      // row stride of the table, a multiple of 32
    int *status;     // nullable: where a bounded wait that gives up is reported
    const unsigned char *tc_cent;   // tensor-core layout of the centroids (bulk path)
    float *gmax;     // nullable: [nq][gld] maxima of each 32-centroid group
    int64_t gld;
    int mode;                // kRankTable, kRankMax or kRankKeep
    const uint32_t *lkey;    // kRankKeep: [nq] threshold keys
    float *keep_s;           // kRankKeep: [nq][nranges][keep_cap] kept scores, per range
    int32_t *keep_i;         //            and their centroid ids, in id order
    int *keep_n;             //            [nq][nranges] how many each range had (even past keep_cap)
    int keep_cap;            //            slots per range
};

// what the ranking contraction's epilogue does with a query's scores:
// store them all (and the group maxima when gmax is set), only the maxima of
// each 32-centroid group, or only the scores that reach the query's threshold
constexpr int kRankTable = 0, kRankMax = 1, kRankKeep = 2;

__device__ int g_rank_status_sink;

struct RankMode {
    using Args = RankArgs;
    static constexpr int kN = 128;
    struct Tile {
        int64_t q0;    // first query
        int ni;
        int64_t c0;    // first centroid of the tile's range
        int64_t nb;    // centroids in the range
    };
    __device__ static int n_ranges(const Args &a) { return (int)ceil_div(a.nlist, kRankRange); }
    __device__ static int num_tiles(const Args &a) { return (int)ceil_div(a.nq, tcp::kM) * n_ranges(a); }
    // every tile costs about the same: a static stride over the blocks
    __device__ static int *tile_counter(const Args &) { return nullptr; }
    __device__ static int d(const Args &a) { return a.d; }
    __device__ static int *status(const Args &a) { return a.status ? a.status : &g_rank_status_sink; }
    __device__ static Tile tile(const Args &a, int t) {
        const int nr = n_ranges(a);
        Tile T;
        T.q0 = (int64_t)(t / nr) * tcp::kM;
        T.ni = (int)(a.nq - T.q0 < tcp::kM ? a.nq - T.q0 : tcp::kM);
        T.c0 = (int64_t)(t % nr) * kRankRange;
        T.nb = a.nlist - T.c0 < kRankRange ? a.nlist - T.c0 : kRankRange;
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
        float *row;      // kRankTable: this query's table row from the range start
        float *grow;     // this query's group maxima from the range start, or nullptr
        float *ks;       // kRankKeep: this query's kept scores / ids for the range
        int32_t *ki;
        int kn;
        int64_t keep_at; // kRankKeep: index of this (query, range) in keep_n
        float thr_raw;   // kRankKeep: the threshold score x 2^16
        __device__ void begin(const Args &a, const Tile &T, int slot, unsigned char *) {
            valid = slot < T.ni;
            const int64_t q = T.q0 + slot;
            row = (valid && a.mode == kRankTable) ? a.scores + q * a.ld + T.c0 : nullptr;
            grow = (valid && a.gmax) ? a.gmax + q * a.gld + T.c0 / 32 : nullptr;
            kn = 0;
            ks = nullptr;
            ki = nullptr;
            thr_raw = 0.f;
            keep_at = 0;
            if (valid && a.mode == kRankKeep) {
                keep_at = q * n_ranges(a) + T.c0 / kRankRange;
                ks = a.keep_s + keep_at * a.keep_cap;
                ki = a.keep_i + keep_at * a.keep_cap;
                thr_raw = key_score(a.lkey[q]) * 65536.f;   // exact: a power-of-two scale
            }
        }
        // v holds the chunk's raw accumulator values: scores x 2^16
        __device__ void chunk(const Args &a, const Tile &T, int64_t col0, const float (&v)[32], int ncol) {
            if (!valid || ncol <= 0) return;
            constexpr float kS = 1.f / 65536.f;
            if (row) {   // ld and the range start are multiples of 32: whole groups fit
                float4 *dst = reinterpret_cast<float4 *>(row + col0);
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    dst[j] = make_float4(v[4 * j] * kS, v[4 * j + 1] * kS, v[4 * j + 2] * kS, v[4 * j + 3] * kS);
            }
            if (grow) {   // the group's maximum over its real columns only
                float mx = v[0];
#pragma unroll
                for (int j = 1; j < 32; ++j) mx = j < ncol ? fmaxf(mx, v[j]) : mx;
                grow[col0 / 32] = mx * kS;
            }
            if (ks) {   // the scores that reach the threshold, in id order
                // (a mask straight from the compares: some lane of a warp
                // nearly always has a candidate in a group, so a maximum
                // test first would not let the warp skip the group)
                unsigned m = 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) m |= v[j] >= thr_raw ? (1u << j) : 0u;
                if (ncol < 32) m &= (1u << ncol) - 1u;
                while (m) {   // counted past keep_cap: an overflow is seen, not lost
                    const int j = __ffs(m) - 1;
                    m &= m - 1u;
                    if (kn < a.keep_cap) {
                        ks[kn] = pick32(v, j) * kS;
                        ki[kn] = (int32_t)(T.c0 + col0 + j);
                    }
                    ++kn;
                }
            }
        }
        __device__ void prefetch(const Args &, const Tile &, int) {}
        __device__ void start(const Args &, const Tile &, int) {}
        __device__ void end(const Args &a, const Tile &) {
            if (ks) a.keep_n[keep_at] = kn;
        }
    };
};
static_assert(kRankRange % RankMode::kN == 0 && kRankRange % kTcRows == 0, "");

__global__ void __launch_bounds__(tcp::kThreads, 1) k_rank_tc(RankArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcp::run_pipeline<RankMode>(a, smem_raw);
}

int rank_bulk_stages(int d) { return tcb::stages_for((int)ceil_div(d, 64), 0, 232448 - 128); }

__global__ void __launch_bounds__(tcb::kThreads, 1) k_rank_bulk(RankArgs a, int stages) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RankMode>(a, smem_raw, stages);
}

constexpr int kSelectWarps = 4;
constexpr int kSelectMaxR = 8;   // lane order statistics used for the lower bracket
constexpr int kStage2 = 16;      // keys per lane of the second selection step (512 entries)
constexpr int kGroupMax = 2048;  // group maxima one threshold warp holds (64 per lane)

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
// given T and C from warp_threshold(key, want, want, ..).  C == want: every
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
                bc[p] = id_of(c);
            }
        }
        pos += __popc(sb);
    }
    __syncwarp();
}

// The want best of the warp's cnt entries into bs/bc[0 .. want-1], in entry
// order (sort_buffer orders them).  With many keys per lane and a second-step
// buffer (ck/ci, 32 * K2 entries; nullable): a first threshold, refined
// until at most 32 * K2 keys reach it (K2 about 2 want / 32), the keys that
// reach it compacted there in entry order, and the exact selection over K2
// keys per lane.
template <int K2, int KPL, class IdOf>
__device__ __forceinline__ bool select_two_step(const uint32_t (&key)[KPL], int cnt, int want,
                                                IdOf id_of, uint32_t *ck, int *ci, float *bs,
                                                int *bc) {
    uint32_t T;
    int C;
    warp_threshold(key, want, 32 * K2, T, C);
    if (C > 32 * K2) {   // T is the want-th largest key itself, tied past the buffer
        warp_gather_exact(key, cnt, want, T, C, id_of, bs, bc);
        return true;
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
            ci[p] = id_of(c);
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
    warp_gather_exact(k2, pos, want, T, C, [&](int c) { return ci[c]; }, bs, bc);
    return true;
}

template <int K2, int KPL, class IdOf>
__device__ __forceinline__ void warp_select_exact(const uint32_t (&key)[KPL], int cnt, int want,
                                                  IdOf id_of, uint32_t *ck, int *ci, float *bs,
                                                  int *bc) {
    static_assert(K2 <= kStage2, "");
    if (want <= 0) return;
    if constexpr (KPL > kStage2) {
        if (ck) {
            select_two_step<K2>(key, cnt, want, id_of, ck, ci, bs, bc);
            return;
        }
    }
    uint32_t T;
    int C;
    warp_threshold(key, want, want, T, C);
    warp_gather_exact(key, cnt, want, T, C, id_of, bs, bc);
}

// One warp per (query, segment of at most kSelectSeg entries).  The
// segment's entries are positions s*seg .. min(M, (s+1)*seg)-1 of the query's
// row of `in_s` (ids from `in_id`, or the position itself when in_id is null),
// in id order among equal scores (a row of centroid scores, or the sorted
// outputs of consecutive id ranges); want = min(nprobe, entries).  Output: the
// want best in order at out_id/out_s[q * out_ld + s * nprobe ..], then
// (-inf, INT32_MAX) padding up to nprobe.  qlist (nullable): only the queries
// qlist[0 .. *qlist_n - 1]; the warps stride over them.  seg_cnt (nullable):
// [nq][nseg] entries actually present in each segment.  nprobe <= 32 * R.
// Eight blocks per SM (64 registers) where the keys fit: the selection is a
// chain of dependent warp reductions, so it needs the warps to hide their
// latency.
template <int KPL, int R>   // entries per lane: seg <= 32 * KPL
__global__ void __launch_bounds__(kSelectWarps * 32, (KPL >= 64 || R >= 8) ? 4 : 8)
    k_select(
    const float *__restrict__ in_s, const int32_t *__restrict__ in_id, int64_t in_ld, int64_t nq,
    int64_t M, int seg, int nseg, int nprobe, int32_t *__restrict__ out_id,
    float *__restrict__ out_s, int64_t out_ld, const int *__restrict__ qlist,
    const int *__restrict__ qlist_n, const int *__restrict__ seg_cnt) {
    extern __shared__ __align__(16) unsigned char sel_smem[];
    // second-step keys per lane: about twice nprobe / 32
    constexpr int kK2 = R <= 2 ? 4 : R == 4 ? 8 : kStage2;
    constexpr int kSort = 32 * R;
    constexpr int kS2 = KPL > kStage2 ? 32 * kK2 : 0;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *bs = reinterpret_cast<float *>(sel_smem) + (size_t)warp * 2 * (kSort + kS2);
    int *bc = reinterpret_cast<int *>(bs + kSort);
    uint32_t *ck = kS2 ? reinterpret_cast<uint32_t *>(bc + kSort) : nullptr;
    int *ci = kS2 ? reinterpret_cast<int *>(ck + kS2) : nullptr;
    const int64_t total = (qlist ? (int64_t)*qlist_n : nq) * nseg;
    for (int64_t w = (int64_t)blockIdx.x * kSelectWarps + warp; w < total;
         w += (int64_t)gridDim.x * kSelectWarps) {
        const int64_t q = qlist ? (int64_t)qlist[w / nseg] : w / nseg;
        const int sg = (int)(w % nseg);
        const int64_t p0 = (int64_t)sg * seg;
        int cnt = (int)(M - p0 < seg ? M - p0 : seg);
        if (seg_cnt && seg_cnt[q * nseg + sg] < cnt) cnt = seg_cnt[q * nseg + sg];
        const int want = nprobe < cnt ? nprobe : cnt;
        const float *row = in_s + q * in_ld + p0;
        const int32_t *rid = in_id ? in_id + q * in_ld + p0 : nullptr;
        uint32_t key[KPL];   // the scores themselves are recovered from the keys
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            const int c = j * 32 + lane;
            key[j] = c < cnt ? order_key(row[c]) : 0u;   // padding ranks below every score
        }
        warp_select_exact<kK2>(key, cnt, want, [&](int c) { return rid ? rid[c] : (int)(p0 + c); },
                               ck, ci, bs, bc);
        sort_buffer<R>(bs, bc, want);
        int32_t *oi = out_id + q * out_ld + (int64_t)sg * nprobe;
        float *os = out_s ? out_s + q * out_ld + (int64_t)sg * nprobe : nullptr;
        for (int p = lane; p < nprobe; p += 32) {
            oi[p] = p < want ? bc[p] : INT32_MAX;
            if (os) os[p] = p < want ? bs[p] : -__int_as_float(0x7f800000);
        }
        __syncwarp();
    }
}

// Threshold from group maxima: one warp per query over its ng maxima of
// 32-centroid groups (ng >= nprobe).  The nprobe-th largest maximum L is a
// score of nprobe different centroids at least, so at least nprobe scores are
// >= L and the nprobe best all are.  Writes the order key of L.
template <int KPL>
__global__ void __launch_bounds__(kSelectWarps * 32) k_group_threshold(
    const float *__restrict__ gmax, int64_t gld, int64_t nq, int ng, int nprobe,
    uint32_t *__restrict__ lkey) {
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
    warp_threshold(key, nprobe, nprobe, T, C);   // refined to the nprobe-th largest
    if (lane == 0) lkey[q] = T;
}

constexpr int kSegCap = 256;        // candidates one table segment may hand on

// One warp per (query, segment of kSelectSeg scores): the scores that reach
// the query's threshold key, in id order, into the segment's kSegCap slots of
// cand_s/cand_i [q][nseg * kSegCap]; their number (even past kSegCap) into
// seg_n[q][nseg].  Lane l reads the segment's 64 scores l*64 .. l*64+63 with
// 16-byte loads, all issued before any is used.
__global__ void __launch_bounds__(kSelectWarps * 32) k_compact_seg(
    const float *__restrict__ scores, int64_t ld, int64_t nq, int64_t nlist, int nseg,
    const uint32_t *__restrict__ lkey, float *__restrict__ cand_s, int32_t *__restrict__ cand_i,
    int *__restrict__ seg_n) {
    constexpr int kPer = kSelectSeg / 32;   // 64 scores per lane
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t w = (int64_t)blockIdx.x * kSelectWarps + warp;
    if (w >= nq * nseg) return;
    const int64_t q = w / nseg;
    const int sg = (int)(w % nseg);
    const int64_t c0 = (int64_t)sg * kSelectSeg + lane * kPer;   // this lane's first column
    const float *row = scores + q * ld;
    const uint32_t L = lkey[q];
    float4 v[kPer / 4];
#pragma unroll
    for (int i = 0; i < kPer / 4; ++i)   // ld is a multiple of 32: a 4-group below ld is whole
        v[i] = c0 + 4 * i < ld ? *reinterpret_cast<const float4 *>(row + c0 + 4 * i)
                               : make_float4(0.f, 0.f, 0.f, 0.f);
    uint64_t hit = 0;   // bit j: column c0 + j qualifies
#pragma unroll
    for (int i = 0; i < kPer / 4; ++i) {
        const float x[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int j = 4 * i + e;
            if (c0 + j < nlist && order_key(x[e]) >= L) hit |= 1ull << j;
        }
    }
    // this lane's place among the segment's candidates: lanes hold consecutive columns
    const int mine = __popcll(hit);
    int x = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    int p = x - mine;
    float *os = cand_s + (q * nseg + sg) * kSegCap;
    int32_t *oi = cand_i + (q * nseg + sg) * kSegCap;
    while (hit) {
        const int j = __ffsll((long long)hit) - 1;
        hit &= hit - 1;
        if (p < kSegCap) {   // the rare candidate's score again (cached), not a register pick
            os[p] = row[c0 + j];
            oi[p] = (int)(c0 + j);
        }
        ++p;
    }
    if (lane == 31) seg_n[q * nseg + sg] = x;
}

// the nprobe best of n candidates (keys ck, ids ci in shared memory, id order;
// n <= 32 * KPL, n >= nprobe) into bs/bc, in id order
template <int KPL>
__device__ __forceinline__ void compact_finish(const uint32_t *ck, const int *ci, int n, int nprobe,
                                               float *bs, int *bc) {
    const int lane = threadIdx.x & 31;
    uint32_t key[KPL];
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        key[j] = c < n ? ck[c] : 0u;
    }
    warp_select_exact<kStage2>(key, n, nprobe, [&](int c) { return ci[c]; }, (uint32_t *)nullptr,
                               (int *)nullptr, bs, bc);
}

// One warp per query: its segments' candidates (at most segcap kept per
// segment) gathered in order (id order) into ccap slots, then the nprobe best
// sorted into order/cscores.  A segment past segcap or more than ccap in all
// (many equal scores): the query is appended to ovf_list (count in *ovf_n,
// zeroed before the launch) and left to an exact fallback.  nprobe <= 32 * R.
template <int R>
__global__ void __launch_bounds__(kSelectWarps * 32, 6) k_compact_final(
    const float *__restrict__ cand_s, const int32_t *__restrict__ cand_i,
    const int *__restrict__ seg_n, int64_t nq, int nseg, int segcap, int nprobe, int ccap,
    int32_t *__restrict__ order, float *__restrict__ cscores, int *__restrict__ ovf_list,
    int *__restrict__ ovf_n) {
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
    // segment counts and their running offsets, 32 segments at a time
    int n = 0;
    bool over = false;
    for (int s0 = 0; s0 < nseg; s0 += 32) {
        const int sg = s0 + lane;
        const int c = sg < nseg ? seg_n[q * nseg + sg] : 0;
        over |= __any_sync(0xffffffffu, c > segcap);
        int x = c;   // inclusive scan over the lanes
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        const int total = __shfl_sync(0xffffffffu, x, 31);
        if (!over && n + total <= ccap && c > 0) {
            // lane l copies segment s0 + l to its place: the segments' loads
            // are in flight together, four of each lane's at a time
            const int at = n + x - c;
            const float *ss = cand_s + (q * nseg + sg) * (int64_t)segcap;
            const int32_t *si = cand_i + (q * nseg + sg) * (int64_t)segcap;
#pragma unroll 4
            for (int i = 0; i < c; ++i) {
                ck[at + i] = order_key(ss[i]);
                ci[at + i] = si[i];
            }
        }
        n += total;
        over |= n > ccap;
    }
    if (over) {
        if (lane == 0) ovf_list[atomicAdd(ovf_n, 1)] = (int)q;
        return;
    }
    __syncwarp();
    // keys per lane sized to the candidates (warp-uniform n)
    if (n <= 128)
        compact_finish<4>(ck, ci, n, nprobe, bs, bc);
    else if (n <= 512)
        compact_finish<16>(ck, ci, n, nprobe, bs, bc);
    else if (n <= 1024)
        compact_finish<32>(ck, ci, n, nprobe, bs, bc);
    else
        compact_finish<64>(ck, ci, n, nprobe, bs, bc);
    sort_buffer<R>(bs, bc, nprobe);
    for (int p = lane; p < nprobe; p += 32) {
        order[q * nprobe + p] = bc[p];
        if (cscores) cscores[q * nprobe + p] = bs[p];
    }
}

// ---------------------------------------------------------------------------
bool rank_tc_supported(int64_t nlist, int nprobe) { return nlist >= 1 && nprobe <= nlist; }

int64_t rank_tc_ld(int64_t nlist) { return round_up(nlist, 32); }

// entries each selection level leaves per query (level 0 = the score row)
static int64_t level_entries(int64_t M, int nprobe) { return ceil_div(M, kSelectSeg) * nprobe; }

// more centroids than one selecting warp holds: a threshold from the maxima
// of 32-centroid groups when there are at least nprobe groups (and few enough
// for one warp), then one compacting pass
static bool use_group_threshold(int64_t nlist, int nprobe) {
    const int64_t ng = ceil_div(nlist, 32);
    return nlist > kSelectSeg && ng >= nprobe && ng <= kGroupMax;
}

// Under the group threshold, narrow rows (d <= 128) skip the score table: one
// contraction writes only the group maxima, a second keeps only the scores
// that reach the threshold.  Two passes of 6d fp16 products per score cost
// less than writing and reading 8 bytes per score when d is this small.
static bool use_two_pass(int64_t nlist, int nprobe, int d) {
    return use_group_threshold(nlist, nprobe) && d <= 128;
}

static int pow2_at_least(int64_t x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

// kept slots per 2,048-centroid range on the two-pass path: four times a
// range's even share of nprobe (the threshold keeps a little over nprobe
// scores in all), at least 64.  A range past it sends its query to the FP32
// fallback.
static int keep_cap(int64_t nlist, int nprobe) {
    const int64_t nseg = ceil_div(nlist, kRankRange);
    const int c = pow2_at_least(ceil_div(4 * (int64_t)nprobe, nseg));
    return (int)std::min<int64_t>(kRankRange, std::max(64, c));
}

// candidates one compacting warp holds: 4 P (P = nprobe rounded up to a
// power of two), between 512 and 2,048
static int compact_cap(int nprobe) {
    return std::min(2048, std::max(512, 4 * pow2_at_least(nprobe)));
}

// registers per lane of the sort of nprobe entries
static int sort_regs(int nprobe) { return std::max(2, pow2_at_least(nprobe) / 32); }

// Scratch of one query, in the order enqueue_rank_tc lays it out:
//   score row (table path only)                      round_up(nlist, 32) f32
//   two level buffers (scores, then ids)             2 x lvl x 8 B   (table path, nlist > kSelectSeg)
//   group maxima                                     round_up(ng, 4) f32
//   candidate slots (scores, then ids)               nseg x cap x 8 B (cap = kSegCap, or
//                                                    keep_cap on the two-pass path)
//   candidate counts, threshold key, overflow list   round_up(nseg, 4) x 4 B + 8 B
// and once per chunk the overflow count (kRankFixedBytes).
constexpr int64_t kRankFixedBytes = 256;
struct RankScratch {
    int64_t ld, lvl, gld, cap;
    int nseg;
    bool table, grouped;
    int64_t per_query() const {
        int64_t b = table ? ld * 4 : 0;
        b += 2 * lvl * 8;
        if (grouped) b += gld * 4 + (int64_t)nseg * cap * 8 + round_up(nseg, 4) * 4 + 8;
        return b;
    }
};

static RankScratch rank_scratch(int64_t nlist, int nprobe, int d) {
    RankScratch r;
    r.ld = rank_tc_ld(nlist);
    r.grouped = use_group_threshold(nlist, nprobe);
    r.table = !use_two_pass(nlist, nprobe, d);
    // the two-pass path falls back to the FP32 ranking, not to the levels
    r.lvl = (nlist > kSelectSeg && r.table) ? round_up(level_entries(nlist, nprobe), 4) : 0;
    r.gld = round_up(ceil_div(nlist, 32), 4);
    r.nseg = (int)ceil_div(nlist, kSelectSeg);
    r.cap = r.table ? kSegCap : keep_cap(nlist, nprobe);
    return r;
}

int64_t rank_tc_chunk(int64_t nq, int64_t nlist, int nprobe, int d) {
    int64_t c = kRankScratchBytes / rank_scratch(nlist, nprobe, d).per_query();
    c = c / tcp::kM * tcp::kM;
    if (c < tcp::kM) c = tcp::kM;
    return nq < c ? nq : c;
}

size_t rank_tc_scratch_bytes(int64_t nq, int64_t nlist, int nprobe, int d) {
    return (size_t)(rank_tc_chunk(nq, nlist, nprobe, d) * rank_scratch(nlist, nprobe, d).per_query() +
                    kRankFixedBytes);
}

static size_t tc_smem() { return tcp::Geometry<RankMode::kN>::smem_bytes(0); }

// shared memory of the selecting kernels (kSelectWarps warps, each with its
// own buffers)
static size_t select_smem(int kpl, int R) {
    const int k2 = R <= 2 ? 4 : R == 4 ? 8 : kStage2;   // k_select's second-step keys per lane
    const size_t s2 = kpl > kStage2 ? 32 * (size_t)k2 : 0;
    return (size_t)kSelectWarps * (32 * (size_t)R + s2) * 8;
}
static size_t compact_smem(int ccap, int R) {
    return (size_t)kSelectWarps * ((size_t)ccap + 32 * (size_t)R) * 8;
}

template <int R>
static cudaError_t set_compact_attr(int ccap) {
    return cudaFuncSetAttribute(k_compact_final<R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)compact_smem(ccap, R));
}

cudaError_t prepare_rank_tc(int nprobe, int d) {
    cudaError_t e = cudaFuncSetAttribute(k_rank_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)tc_smem());
    const int bulk = rank_bulk_stages(d);
    if (e == cudaSuccess && bulk)
        e = cudaFuncSetAttribute(k_rank_bulk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)tcb::smem_bytes(bulk, 0));
    // the selections stay below the 48 KB default; the compacting warps may not
    const int ccap = compact_cap(nprobe);
    if (e == cudaSuccess) e = set_compact_attr<2>(ccap);
    if (e == cudaSuccess) e = set_compact_attr<4>(ccap);
    if (e == cudaSuccess) e = set_compact_attr<8>(ccap);
    if (e == cudaSuccess) e = set_compact_attr<16>(ccap);
    // the two-pass path's exact fallback
    if (e == cudaSuccess && d <= 128) e = prepare_rank(nprobe);
    return e;
}

template <int KPL>
static void select_r(int R, dim3 grid, size_t smem, cudaStream_t st, const float *in_s,
                     const int32_t *in_id, int64_t in_ld, int64_t nq, int64_t M, int seg, int nseg,
                     int nprobe, int32_t *out_id, float *out_s, int64_t out_ld, const int *qlist,
                     const int *qlist_n, const int *seg_cnt) {
#define SIEVE_SELECT(RR)                                                                        \
    k_select<KPL, RR><<<grid, kSelectWarps * 32, smem, st>>>(in_s, in_id, in_ld, nq, M, seg, nseg, \
                                                             nprobe, out_id, out_s, out_ld, qlist, \
                                                             qlist_n, seg_cnt)
    switch (R) {
        case 2: SIEVE_SELECT(2); break;
        case 4: SIEVE_SELECT(4); break;
        case 8: SIEVE_SELECT(8); break;
        default: SIEVE_SELECT(16); break;
    }
#undef SIEVE_SELECT
}

// one selection level: the best nprobe of every segment of at most kSelectSeg
// entries (nseg = 1: the final order).  qlist/qlist_n (nullable, device): only
// the listed queries, on a grid of a few blocks per SM that strides over them.
static void launch_select(const float *in_s, const int32_t *in_id, int64_t in_ld, int64_t nq,
                          int64_t M, int nprobe, int32_t *out_id, float *out_s, int64_t out_ld,
                          const int *qlist, const int *qlist_n, const int *seg_cnt, cudaStream_t st) {
    const int seg = M < kSelectSeg ? (int)M : kSelectSeg;
    const int nseg = (int)ceil_div(M, kSelectSeg);
    const int R = sort_regs(nprobe);
    int64_t blocks = ceil_div(nq * nseg, kSelectWarps);
    if (qlist) blocks = std::min<int64_t>(blocks, 4 * (int64_t)num_sms());
    const dim3 grid((unsigned)blocks);
    const int kpl = std::max(4, pow2_at_least(ceil_div(seg, 32)));
#define SIEVE_SEL_K(K)                                                                          \
    select_r<K>(R, grid, select_smem(K, R), st, in_s, in_id, in_ld, nq, M, seg, nseg, nprobe,     \
                out_id, out_s, out_ld, qlist, qlist_n, seg_cnt)
    if (kpl <= 4)
        SIEVE_SEL_K(4);
    else if (kpl <= 16)
        SIEVE_SEL_K(16);
    else if (kpl <= 32)
        SIEVE_SEL_K(32);
    else
        SIEVE_SEL_K(64);
#undef SIEVE_SEL_K
}

static void launch_compact_final(const float *cand_s, const int32_t *cand_i, const int *seg_n,
                                 int64_t nq, int nseg, int segcap, int nprobe, int32_t *order,
                                 float *cscores, int *ovf_list, int *ovf_n, cudaStream_t st) {
    const unsigned blocks = (unsigned)ceil_div(nq, kSelectWarps);
    const int ccap = compact_cap(nprobe);
#define SIEVE_COMPACT(RR)                                                                      \
    k_compact_final<RR><<<blocks, kSelectWarps * 32, compact_smem(ccap, RR), st>>>(               \
        cand_s, cand_i, seg_n, nq, nseg, segcap, nprobe, ccap, order, cscores, ovf_list, ovf_n)
    switch (sort_regs(nprobe)) {
        case 2: SIEVE_COMPACT(2); break;
        case 4: SIEVE_COMPACT(4); break;
        case 8: SIEVE_COMPACT(8); break;
        default: SIEVE_COMPACT(16); break;
    }
#undef SIEVE_COMPACT
}

int rank_tc_launches(int64_t nq, int64_t nlist, int nprobe, int d) {
    if (nq <= 0) return 0;
    int per;
    if (use_two_pass(nlist, nprobe, d)) {
        per = 5;   // maxima pass, threshold, keeping pass, final warps, FP32 fallback
    } else {
        per = 2;   // contraction, final selection level
        if (use_group_threshold(nlist, nprobe)) per += 3;   // threshold, compaction, final warps
        for (int64_t M = nlist; M > kSelectSeg; M = level_entries(M, nprobe)) ++per;
    }
    return (int)ceil_div(nq, rank_tc_chunk(nq, nlist, nprobe, d)) * per;
}

int rank_tc_mma_launches(int64_t nq, int64_t nlist, int nprobe, int d) {
    if (nq <= 0) return 0;
    return (int)ceil_div(nq, rank_tc_chunk(nq, nlist, nprobe, d)) *
           (use_two_pass(nlist, nprobe, d) ? 2 : 1);
}

cudaError_t enqueue_rank_tc(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                            int nprobe, int32_t *order, float *cscores, float *scratch, int *status,
                            cudaStream_t st, const unsigned char *tc_cent, float *mma_ms) {
    struct Events {   // mma_ms: a pair per contraction launch, destroyed on every return
        std::vector<cudaEvent_t> v;
        ~Events() {
            for (cudaEvent_t e : v) cudaEventDestroy(e);
        }
    } ev_hold;
    std::vector<cudaEvent_t> &evs = ev_hold.v;
    const int bulk_stages = tc_cent ? rank_bulk_stages(d) : 0;
    const RankScratch L = rank_scratch(nlist, nprobe, d);
    const int64_t chunk = rank_tc_chunk(nq, nlist, nprobe, d);
    // carve the chunk's scratch (RankScratch's order, each part [chunk][...])
    float *p = scratch;
    float *table = p;
    p += L.table ? chunk * L.ld : 0;
    float *cand_s[2];
    int32_t *cand_id[2];
    for (int b = 0; b < 2; ++b) {
        cand_s[b] = p;
        cand_id[b] = reinterpret_cast<int32_t *>(p + chunk * L.lvl);
        p += 2 * chunk * L.lvl;
    }
    float *gmax = p;
    p += L.grouped ? chunk * L.gld : 0;
    float *slot_s = p;
    int32_t *slot_i = reinterpret_cast<int32_t *>(p + chunk * L.nseg * L.cap);
    p += L.grouped ? 2 * chunk * L.nseg * L.cap : 0;
    int *slot_n = reinterpret_cast<int *>(p);
    uint32_t *lkey = reinterpret_cast<uint32_t *>(slot_n + (L.grouped ? chunk * round_up(L.nseg, 4) : 0));
    int *ovf = reinterpret_cast<int *>(lkey + (L.grouped ? chunk : 0));   // [chunk] overflow list
    int *ovf_n = reinterpret_cast<int *>(reinterpret_cast<unsigned char *>(scratch) +
                                         chunk * L.per_query());       // its count
    const int ng = (int)ceil_div(nlist, 32);
    for (int64_t q0 = 0; q0 < nq; q0 += chunk) {
        const int64_t n = nq - q0 < chunk ? nq - q0 : chunk;
        const int tiles = (int)(ceil_div(n, tcp::kM) * ceil_div(nlist, kRankRange));
        auto contract = [&](const RankArgs &a) {
            if (mma_ms) {
                evs.resize(evs.size() + 2);
                cudaEventCreate(&evs[evs.size() - 2]);
                cudaEventCreate(&evs.back());
                cudaEventRecord(evs[evs.size() - 2], st);
            }
            if (bulk_stages)
                k_rank_bulk<<<std::min(tiles, num_sms()), tcb::kThreads,
                              tcb::smem_bytes(bulk_stages, 0), st>>>(a, bulk_stages);
            else
                k_rank_tc<<<std::min(tiles, num_sms()), tcp::kThreads, tc_smem(), st>>>(a);
            if (mma_ms) cudaEventRecord(evs.back(), st);
        };
        RankArgs a{Q + q0 * d, n, C, nlist, d, table, L.ld, status, tc_cent,
                   L.grouped ? gmax : nullptr, L.gld, L.table ? kRankTable : kRankMax,
                   lkey, slot_s, slot_i, slot_n, (int)L.cap};
        contract(a);
        int32_t *o = order + q0 * nprobe;
        float *cs = cscores ? cscores + q0 * nprobe : nullptr;
        const int *qlist = nullptr, *qlist_n = nullptr;
        if (L.grouped) {
            const unsigned wblocks = (unsigned)ceil_div(n, kSelectWarps);
            const int kpl = pow2_at_least(ceil_div(ng, 32));
#define SIEVE_GTHR(K)                                                                              \
    k_group_threshold<K><<<wblocks, kSelectWarps * 32, 0, st>>>(gmax, L.gld, n, ng, nprobe, lkey)
            switch (kpl) {
                case 1: SIEVE_GTHR(1); break;
                case 2: SIEVE_GTHR(2); break;
                case 4: SIEVE_GTHR(4); break;
                case 8: SIEVE_GTHR(8); break;
                case 16: SIEVE_GTHR(16); break;
                case 32: SIEVE_GTHR(32); break;
                default: SIEVE_GTHR(64); break;
            }
#undef SIEVE_GTHR
            if (L.table) {
                k_compact_seg<<<(unsigned)ceil_div(n * L.nseg, kSelectWarps), kSelectWarps * 32, 0,
                                st>>>(table, L.ld, n, nlist, L.nseg, lkey, slot_s, slot_i, slot_n);
            } else {
                RankArgs keep = a;   // the second contraction keeps what reaches the threshold
                keep.gmax = nullptr;
                keep.mode = kRankKeep;
                contract(keep);
            }
            cudaError_t e = cudaMemsetAsync(ovf_n, 0, sizeof(int), st);
            if (e != cudaSuccess) return e;
            launch_compact_final(slot_s, slot_i, slot_n, n, L.nseg, (int)L.cap, nprobe, o, cs, ovf,
                                 ovf_n, st);
            if (!L.table) {
                // the queries whose kept slots overflowed: the FP32 ranking, exact
                e = enqueue_rank(Q + q0 * d, n, C, nlist, d, nprobe, o, cs, st, ovf, ovf_n);
                if (e != cudaSuccess) return e;
                e = cudaGetLastError();
                if (e != cudaSuccess) return e;
                continue;
            }
            qlist = ovf;   // the levels below run only for the overflowing queries
            qlist_n = ovf_n;
        }
        // levels over the score table until one segment is left
        const float *in_s = table;
        const int32_t *in_id = nullptr;
        int64_t in_ld = L.ld, M = nlist;
        int buf = 0;
        while (M > kSelectSeg) {
            launch_select(in_s, in_id, in_ld, n, M, nprobe, cand_id[buf], cand_s[buf], L.lvl, qlist,
                          qlist_n, nullptr, st);
            in_s = cand_s[buf];
            in_id = cand_id[buf];
            in_ld = L.lvl;
            M = level_entries(M, nprobe);
            buf ^= 1;
        }
        launch_select(in_s, in_id, in_ld, n, M, nprobe, o, cs, nprobe, qlist, qlist_n, nullptr, st);
        cudaError_t e = cudaGetLastError();
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
