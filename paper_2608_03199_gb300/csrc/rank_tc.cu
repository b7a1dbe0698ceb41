// rank_tc.cu -- centroid ranking on the tcgen05 tensor cores (Sec. 2.3,
// Sec. 4.1: P_i = the nprobe centroids with the largest inner product with
// q_i, best first, equal scores by lower centroid id), for any nlist.
//
// Per chunk of queries:
//   k_rank_bulk / k_rank_tc  the tensor-core contraction (tc_bulk.cuh with the
//              centroids' tensor-core layout, else the converter pipeline of
//              tc_pipeline.cuh): a tile is 128 consecutive queries (A rows)
//              against one range of kRankRange centroids (B rows, 128 per
//              chunk); each epilogue thread stores its query's scores into a
//              score table [queries][ld] in the caller's workspace
//   k_select   one warp per (query, segment of at most kSelectSeg entries):
//              the segment's best min(nprobe, size) entries, sorted by
//              (score desc, id asc).  With nlist <= kSelectSeg one segment
//              gives the order directly; otherwise each level keeps the best
//              nprobe of every segment (the nprobe best of a set lie among the
//              nprobe best of each of its parts) until one segment is left.
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
    float *keep_s;           // kRankKeep: [nq][nranges][kRankRange] kept scores, per range
    int32_t *keep_i;         //            and their centroid ids, in id order
    int *keep_n;             //            [nq][nranges] how many each range kept
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
                ks = a.keep_s + keep_at * kRankRange;
                ki = a.keep_i + keep_at * kRankRange;
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
                float mx[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) mx[j] = fmaxf(v[j], v[j + 16]);
#pragma unroll
                for (int w = 8; w > 0; w >>= 1)
#pragma unroll
                    for (int j = 0; j < w; ++j) mx[j] = fmaxf(mx[j], mx[j + w]);
                if (!(mx[0] >= thr_raw)) return;
                unsigned m = 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) m |= (v[j] >= thr_raw && j < ncol) ? (1u << j) : 0u;
                while (m) {   // at most kRankRange per range: the slots cannot overflow
                    const int j = __ffs(m) - 1;
                    m &= m - 1u;
                    ks[kn] = pick32(v, j) * kS;
                    ki[kn] = (int32_t)(T.c0 + col0 + j);
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
constexpr int kSelectSmallC = 4; // candidate keys per lane of the two-step selection (P <= 64)

// warp-wide reductions in one instruction (redux.sync), not a chain of shuffles
__device__ __forceinline__ int warp_sum(int x) { return __reduce_add_sync(0xffffffffu, x); }

template <int KPL>
__device__ __forceinline__ int count_ge(const uint32_t (&key)[KPL], uint32_t t) {
    int c = 0;
#pragma unroll
    for (int j = 0; j < KPL; ++j) c += key[j] >= t;
    return warp_sum(c);
}

// A threshold T <= T* (T* = the want-th largest of the warp's keys; keys of
// padding are 0, below every score) with C = #{keys >= T} >= want, refined
// bit by bit (the largest T with at least want keys >= T) until C <= cap or
// T == T*.  The search starts from the common high bits of a bracket
// L <= T* <= U: U = the largest key, L = the smallest over lanes of each
// lane's ceil(want / 32)-th largest key (at least want keys are >= L).
template <int KPL>
__device__ __forceinline__ void warp_threshold(const uint32_t (&key)[KPL], int want, int cap,
                                               uint32_t &T, int &C) {
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
    uint32_t U = m[0];
    uint32_t L = 0u;   // r > kSelectMaxR: no lower bracket
#pragma unroll
    for (int i = 0; i < kSelectMaxR; ++i) L = r == i + 1 ? m[i] : L;
    U = __reduce_max_sync(0xffffffffu, U);
    L = __reduce_min_sync(0xffffffffu, L);
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

// The want best of the warp's cnt entries (entry c = key[c / 32] of lane
// c % 32; its id from id_of(c)), sorted by (score desc, id asc) into bs/bc,
// given T and C from warp_threshold.  C <= cap: every key >= T is a candidate;
// otherwise T == T* and the keys > T* plus the first keys equal to it in entry
// order are taken, which are the lowest ids when entry order is id order among
// equal scores.  bs/bc hold 2P >= cap entries; returns the count sorted.
template <int KPL, class IdOf>
__device__ __forceinline__ void warp_gather_sort(const uint32_t (&key)[KPL], int cnt, int want,
                                                 uint32_t T, int C, int cap, IdOf id_of,
                                                 float *bs, int *bc) {
    const int lane = threadIdx.x & 31;
    const unsigned below = (1u << lane) - 1u;
    int pos = 0;
    // the buffer holds cap entries: C <= cap, or exactly want <= cap taken
    // below; the bound on p only keeps a broken invariant from writing past it
    if (C <= cap) {
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            const int c = j * 32 + lane;
            const bool sel = key[j] >= T && c < cnt;
            const unsigned sb = __ballot_sync(0xffffffffu, sel);
            if (sel) {
                const int p = pos + __popc(sb & below);
                if (p < cap) {
                    bs[p] = key_score(key[j]);
                    bc[p] = id_of(c);
                }
            }
            pos += __popc(sb);
        }
    } else {
        int gt = 0;
#pragma unroll
        for (int j = 0; j < KPL; ++j) gt += key[j] > T;
        const int ties_wanted = want - warp_sum(gt);   // >= 1
        int ties_seen = 0;
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            const int c = j * 32 + lane;
            const bool tie = key[j] == T && c < cnt;
            const unsigned tb = __ballot_sync(0xffffffffu, tie);
            const bool sel = key[j] > T || (tie && ties_seen + __popc(tb & below) < ties_wanted);
            const unsigned sb = __ballot_sync(0xffffffffu, sel);
            if (sel) {
                const int p = pos + __popc(sb & below);
                if (p < cap) {
                    bs[p] = key_score(key[j]);
                    bc[p] = id_of(c);
                }
            }
            pos += __popc(sb);
            ties_seen += __popc(tb);
        }
    }
    if (pos > cap) pos = cap;
    int S = 1;   // sort size: a power of two >= pos (pos <= cap)
    while (S < pos) S <<= 1;
    for (int p = pos + lane; p < S; p += 32) {
        bs[p] = -__int_as_float(0x7f800000);
        bc[p] = INT32_MAX;
    }
    __syncwarp();
    if (S <= 64) {
        // bitonic sort in registers: entry i = r * 32 + lane in register r;
        // partners across lanes by shuffles, across registers (j = 32) in place
        const float ninf = -__int_as_float(0x7f800000);
        float s0 = lane < S ? bs[lane] : ninf, s1 = lane + 32 < S ? bs[lane + 32] : ninf;
        int c0 = lane < S ? bc[lane] : INT32_MAX, c1 = lane + 32 < S ? bc[lane + 32] : INT32_MAX;
        for (int k = 2; k <= S; k <<= 1) {
            for (int j = k >> 1; j > 0; j >>= 1) {
                if (j == 32) {   // k == 64: entry lane (kept better) against lane + 32
                    if (ranks_before(s1, c1, s0, c0)) {
                        const float ts = s0;
                        const int tc = c0;
                        s0 = s1;
                        c0 = c1;
                        s1 = ts;
                        c1 = tc;
                    }
                    continue;
                }
                const float ps0 = __shfl_xor_sync(0xffffffffu, s0, j);
                const int pc0 = __shfl_xor_sync(0xffffffffu, c0, j);
                const float ps1 = __shfl_xor_sync(0xffffffffu, s1, j);
                const int pc1 = __shfl_xor_sync(0xffffffffu, c1, j);
                const bool lower = (lane & j) == 0;
                // the lower entry of a pair keeps the better one when its
                // block sorts first-ranked first ((i & k) == 0), else the worse
                const bool take0 = (lower == ((lane & k) == 0)) == ranks_before(ps0, pc0, s0, c0);
                const bool take1 = (lower == (((lane + 32) & k) == 0)) == ranks_before(ps1, pc1, s1, c1);
                if (take0) { s0 = ps0; c0 = pc0; }
                if (take1) { s1 = ps1; c1 = pc1; }
            }
        }
        __syncwarp();
        if (lane < S) { bs[lane] = s0; bc[lane] = c0; }
        if (lane + 32 < S) { bs[lane + 32] = s1; bc[lane + 32] = c1; }
        __syncwarp();
        return;
    }
    // bitonic sort of S entries, first-ranked first
    for (int k = 2; k <= S; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = lane; i < S / 2; i += 32) {
                const int lo = 2 * i - (i & (j - 1));
                const int hi = lo + j;
                const bool up = (lo & k) == 0;
                const float s0 = bs[lo], s1 = bs[hi];
                const int c0 = bc[lo], c1 = bc[hi];
                if (ranks_before(s1, c1, s0, c0) == up) {
                    bs[lo] = s1;
                    bc[lo] = c1;
                    bs[hi] = s0;
                    bc[hi] = c0;
                }
            }
            __syncwarp();
        }
    }
}

// One warp per (query, segment).  The segment's entries are positions
// s*seg .. min(M, (s+1)*seg)-1 of the query's row of `in_s` (ids from `in_id`,
// or the position itself when in_id is null), in id order among equal scores
// (a row of centroid scores, or the sorted outputs of consecutive id ranges);
// want = min(nprobe, entries).  Output: the want best in order at
// out_id/out_s[q * out_ld + s * nprobe ..], then (-inf, INT32_MAX) padding up
// to nprobe.  `only` (nullable): queries with only[q] == 0 are skipped.
// `seg_cnt` (nullable): [nq][nseg] entries actually present in each segment.
// P: a power of two >= nprobe; the sort buffer holds 2P entries.
// Eight blocks per SM (64 registers) where the keys fit: the selection is a chain
// of dependent warp reductions, so it needs the warps to hide their latency
// (timed 25% faster than 120 registers at four blocks).
template <int KPL>   // entries per lane: seg <= 32 * KPL
__global__ void __launch_bounds__(kSelectWarps * 32, KPL >= 64 ? 4 : 8) k_select(
    const float *__restrict__ in_s, const int32_t *__restrict__ in_id, int64_t in_ld, int64_t nq,
    int64_t M, int seg, int nseg, int nprobe, int P, int32_t *__restrict__ out_id,
    float *__restrict__ out_s, int64_t out_ld, const int *__restrict__ only,
    const int *__restrict__ seg_cnt) {
    extern __shared__ __align__(16) unsigned char sel_smem[];
    const int cap = 2 * P;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *bs = reinterpret_cast<float *>(sel_smem) + warp * 2 * cap;   // cap scores, then cap ids
    int *bc = reinterpret_cast<int *>(bs + cap);
    const int64_t w = (int64_t)blockIdx.x * kSelectWarps + warp;
    if (w >= nq * nseg) return;
    const int64_t q = w / nseg;
    if (only && only[q] == 0) return;
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
    uint32_t T;
    int C;
    warp_threshold(key, want, cap, T, C);
    if (C <= cap && cap <= 32 * kSelectSmallC) {
        // two steps: the C candidates (key >= T) go to shared memory in id
        // order, come back as kSelectSmallC keys per lane, and a second, cheap
        // threshold over them leaves exactly want entries to sort
        const unsigned below = (1u << lane) - 1u;
        uint32_t *ck = reinterpret_cast<uint32_t *>(bs);
        int pos = 0;
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            const int c = j * 32 + lane;
            const bool sel = key[j] >= T && c < cnt;
            const unsigned sb = __ballot_sync(0xffffffffu, sel);
            if (sel) {
                const int p = pos + __popc(sb & below);
                if (p < cap) {   // pos <= C <= cap
                    ck[p] = key[j];
                    bc[p] = rid ? rid[c] : (int)(p0 + c);
                }
            }
            pos += __popc(sb);
        }
        __syncwarp();
        uint32_t k2[kSelectSmallC];
        int i2[kSelectSmallC];
#pragma unroll
        for (int j = 0; j < kSelectSmallC; ++j) {
            const int c = j * 32 + lane;
            k2[j] = c < pos ? ck[c] : 0u;
            i2[j] = c < pos ? bc[c] : 0;
        }
        __syncwarp();
        uint32_t T2;
        int C2;
        warp_threshold(k2, want, want, T2, C2);
        warp_gather_sort(k2, pos, want, T2, C2, want, [&](int c) {
            // id of candidate c: held by lane c % 32 in slot c / 32 (c is this lane's)
            int id = i2[0];
#pragma unroll
            for (int j = 1; j < kSelectSmallC; ++j) id = (c >> 5) == j ? i2[j] : id;
            return id;
        }, bs, bc);
    } else {
        warp_gather_sort(key, cnt, want, T, C, cap,
                         [&](int c) { return rid ? rid[c] : (int)(p0 + c); }, bs, bc);
    }
    int32_t *oi = out_id + q * out_ld + (int64_t)sg * nprobe;
    float *os = out_s ? out_s + q * out_ld + (int64_t)sg * nprobe : nullptr;
    for (int p = lane; p < nprobe; p += 32) {
        oi[p] = p < want ? bc[p] : INT32_MAX;
        if (os) os[p] = p < want ? bs[p] : -__int_as_float(0x7f800000);
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

constexpr int kCompactCap = 2048;   // candidates the final warp of a query keeps (64 per lane)
constexpr int kSegCap = 256;        // candidates one segment may hand on

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
// n <= 32 * KPL, n >= nprobe), sorted into bs/bc
template <int KPL>
__device__ __forceinline__ void compact_finish(const uint32_t *ck, const int *ci, int n, int nprobe,
                                               int cap, float *bs, int *bc) {
    const int lane = threadIdx.x & 31;
    uint32_t key[KPL];
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        key[j] = c < n ? ck[c] : 0u;
    }
    uint32_t T;
    int C;
    warp_threshold(key, nprobe, cap, T, C);
    warp_gather_sort(key, n, nprobe, T, C, cap, [&](int c) { return ci[c]; }, bs, bc);
}

// One warp per query: its segments' candidates gathered in order (id order),
// then the nprobe best sorted into order/cscores.  A segment past kSegCap or
// more than kCompactCap in all (many equal scores): the query is flagged in
// ovf and left to the level-by-level selection.
__global__ void __launch_bounds__(kSelectWarps * 32) k_compact_final(
    const float *__restrict__ cand_s, const int32_t *__restrict__ cand_i,
    const int *__restrict__ seg_n, int64_t nq, int nseg, int segcap, int nprobe, int P,
    int32_t *__restrict__ order, float *__restrict__ cscores, int *__restrict__ ovf) {
    extern __shared__ __align__(16) unsigned char sel_smem[];
    const int cap = 2 * P;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char *wbase = sel_smem + (size_t)warp * (kCompactCap * 8 + 2 * cap * 4);
    uint32_t *ck = reinterpret_cast<uint32_t *>(wbase);              // candidate keys
    int *ci = reinterpret_cast<int *>(wbase + kCompactCap * 4);      // candidate ids
    float *bs = reinterpret_cast<float *>(wbase + kCompactCap * 8);  // sort buffer
    int *bc = reinterpret_cast<int *>(bs + cap);
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
        if (!over && n + total <= kCompactCap) {
            // copy each segment's candidates to its place (lanes of the warp in turn)
            for (int t = 0; t < 32 && s0 + t < nseg; ++t) {
                const int ct = __shfl_sync(0xffffffffu, c, t);
                const int at = n + __shfl_sync(0xffffffffu, x, t) - ct;
                const float *ss = cand_s + (q * nseg + s0 + t) * (int64_t)segcap;
                const int32_t *si = cand_i + (q * nseg + s0 + t) * (int64_t)segcap;
                for (int i = lane; i < ct; i += 32) {
                    ck[at + i] = order_key(ss[i]);
                    ci[at + i] = si[i];
                }
            }
        }
        n += total;
        over |= n > kCompactCap;
    }
    if (over) {
        if (lane == 0) ovf[q] = 1;
        return;
    }
    if (lane == 0) ovf[q] = 0;
    __syncwarp();
    // keys per lane sized to the candidates (warp-uniform n)
    if (n <= 256)
        compact_finish<8>(ck, ci, n, nprobe, cap, bs, bc);
    else if (n <= 512)
        compact_finish<16>(ck, ci, n, nprobe, cap, bs, bc);
    else if (n <= 1024)
        compact_finish<32>(ck, ci, n, nprobe, cap, bs, bc);
    else
        compact_finish<kCompactCap / 32>(ck, ci, n, nprobe, cap, bs, bc);
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
    return nlist > kSelectSeg && ng >= nprobe && ng <= kCompactCap;
}

// Under the group threshold, narrow rows (d <= 128) skip the score table: one
// contraction writes only the group maxima, a second keeps only the scores
// that reach the threshold.  Two passes of 6d fp16 products per score cost
// less than writing and reading 8 bytes per score when d is this small.
static bool use_two_pass(int64_t nlist, int nprobe, int d) {
    return use_group_threshold(nlist, nprobe) && d <= 128;
}

// Scratch of one query, in the order enqueue_rank_tc lays it out:
//   score row (table path only)                      round_up(nlist, 32) f32
//   two level buffers (scores, then ids)             2 x lvl x 8 B   (nlist > kSelectSeg)
//   group maxima                                     round_up(ng, 4) f32
//   candidate slots (scores, then ids)               nseg x cap x 8 B (cap = kSegCap, or
//                                                    kRankRange on the two-pass path)
//   candidate counts, threshold key, overflow flag   round_up(nseg, 4) x 4 B + 8 B
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
    r.lvl = nlist > kSelectSeg ? round_up(level_entries(nlist, nprobe), 4) : 0;
    r.grouped = use_group_threshold(nlist, nprobe);
    r.table = !use_two_pass(nlist, nprobe, d);
    r.gld = round_up(ceil_div(nlist, 32), 4);
    r.nseg = (int)ceil_div(nlist, kSelectSeg);
    r.cap = r.table ? kSegCap : kRankRange;
    return r;
}

int64_t rank_tc_chunk(int64_t nq, int64_t nlist, int nprobe, int d) {
    int64_t c = kRankScratchBytes / rank_scratch(nlist, nprobe, d).per_query();
    c = c / tcp::kM * tcp::kM;
    if (c < tcp::kM) c = tcp::kM;
    return nq < c ? nq : c;
}

size_t rank_tc_scratch_bytes(int64_t nq, int64_t nlist, int nprobe, int d) {
    return (size_t)(rank_tc_chunk(nq, nlist, nprobe, d) * rank_scratch(nlist, nprobe, d).per_query());
}

static size_t tc_smem() { return tcp::Geometry<RankMode::kN>::smem_bytes(0); }

static int pow2_at_least(int64_t x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

static size_t select_smem(int P) { return (size_t)kSelectWarps * 2 * (2 * P) * 4; }
static size_t compact_smem(int P) {
    return (size_t)kSelectWarps * ((size_t)kCompactCap * 8 + 2 * (2 * P) * 4);
}

template <int KPL>
static cudaError_t set_select_attr(int P) {
    return cudaFuncSetAttribute(k_select<KPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)select_smem(P));
}

cudaError_t prepare_rank_tc(int nprobe, int d) {
    cudaError_t e = cudaFuncSetAttribute(k_rank_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)tc_smem());
    const int bulk = rank_bulk_stages(d);
    if (e == cudaSuccess && bulk)
        e = cudaFuncSetAttribute(k_rank_bulk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)tcb::smem_bytes(bulk, 0));
    const int P = pow2_at_least(nprobe);
    if (e == cudaSuccess) e = set_select_attr<1>(P);
    if (e == cudaSuccess) e = set_select_attr<2>(P);
    if (e == cudaSuccess) e = set_select_attr<4>(P);
    if (e == cudaSuccess) e = set_select_attr<8>(P);
    if (e == cudaSuccess) e = set_select_attr<16>(P);
    if (e == cudaSuccess) e = set_select_attr<32>(P);
    if (e == cudaSuccess) e = set_select_attr<64>(P);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_compact_final, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)compact_smem(P));
    return e;
}

// one selection level: the best nprobe of every segment of at most kSelectSeg
// entries (nseg = 1: the final order)
static void launch_select(const float *in_s, const int32_t *in_id, int64_t in_ld, int64_t nq,
                          int64_t M, int nprobe, int32_t *out_id, float *out_s, int64_t out_ld,
                          const int *only, const int *seg_cnt, cudaStream_t st) {
    const int seg = M < kSelectSeg ? (int)M : kSelectSeg;
    const int nseg = (int)ceil_div(M, kSelectSeg);
    const int P = pow2_at_least(nprobe);
    const unsigned blocks = (unsigned)ceil_div(nq * nseg, kSelectWarps);
    const size_t smem = select_smem(P);
    const int kpl = pow2_at_least(ceil_div(seg, 32));
#define SIEVE_SELECT(K)                                                                            \
    k_select<K><<<blocks, kSelectWarps * 32, smem, st>>>(in_s, in_id, in_ld, nq, M, seg, nseg,     \
                                                        nprobe, P, out_id, out_s, out_ld, only, \
                                                        seg_cnt)
    switch (kpl) {
        case 1: SIEVE_SELECT(1); break;
        case 2: SIEVE_SELECT(2); break;
        case 4: SIEVE_SELECT(4); break;
        case 8: SIEVE_SELECT(8); break;
        case 16: SIEVE_SELECT(16); break;
        case 32: SIEVE_SELECT(32); break;
        default: SIEVE_SELECT(64); break;
    }
#undef SIEVE_SELECT
}

int rank_tc_launches(int64_t nq, int64_t nlist, int nprobe, int d) {
    if (nq <= 0) return 0;
    int per = 2;                                           // contraction + final selection
    if (use_group_threshold(nlist, nprobe)) per += 3;      // threshold, compaction, gather
    // the two-pass path trades the compaction pass for a second contraction: same count
    for (int64_t M = nlist; M > kSelectSeg; M = level_entries(M, nprobe)) ++per;
    return (int)ceil_div(nq, rank_tc_chunk(nq, nlist, nprobe, d)) * per;
}

cudaError_t enqueue_rank_tc(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                            int nprobe, int32_t *order, float *cscores, float *scratch, int *status,
                            cudaStream_t st, const unsigned char *tc_cent) {
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
    p += chunk * L.gld;
    float *slot_s = p;
    int32_t *slot_i = reinterpret_cast<int32_t *>(p + chunk * L.nseg * L.cap);
    p += 2 * chunk * L.nseg * L.cap;
    int *slot_n = reinterpret_cast<int *>(p);
    uint32_t *lkey = reinterpret_cast<uint32_t *>(slot_n + chunk * round_up(L.nseg, 4));
    int *ovf = reinterpret_cast<int *>(lkey + chunk);
    const int ng = (int)ceil_div(nlist, 32);
    const int P = pow2_at_least(nprobe);
    for (int64_t q0 = 0; q0 < nq; q0 += chunk) {
        const int64_t n = nq - q0 < chunk ? nq - q0 : chunk;
        const int tiles = (int)(ceil_div(n, tcp::kM) * ceil_div(nlist, kRankRange));
        auto contract = [&](const RankArgs &a) {
            if (bulk_stages)
                k_rank_bulk<<<std::min(tiles, num_sms()), tcb::kThreads,
                              tcb::smem_bytes(bulk_stages, 0), st>>>(a, bulk_stages);
            else
                k_rank_tc<<<std::min(tiles, num_sms()), tcp::kThreads, tc_smem(), st>>>(a);
        };
        RankArgs a{Q + q0 * d, n, C, nlist, d, table, L.ld, status, tc_cent,
                   L.grouped ? gmax : nullptr, L.gld, L.table ? kRankTable : kRankMax,
                   lkey, slot_s, slot_i, slot_n};
        contract(a);
        int32_t *o = order + q0 * nprobe;
        float *cs = cscores ? cscores + q0 * nprobe : nullptr;
        const int *only = nullptr;
        const float *lvl0_s = table;       // what the first selection level reads
        const int32_t *lvl0_id = nullptr;
        int64_t lvl0_ld = L.ld;
        const int *lvl0_cnt = nullptr;
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
                // an overflowing query's levels read its kept scores, range by range
                lvl0_s = slot_s;
                lvl0_id = slot_i;
                lvl0_ld = (int64_t)L.nseg * L.cap;
                lvl0_cnt = slot_n;
            }
            k_compact_final<<<wblocks, kSelectWarps * 32, compact_smem(P), st>>>(
                slot_s, slot_i, slot_n, n, L.nseg, (int)L.cap, nprobe, P, o, cs, ovf);
            only = ovf;   // the levels below run only for overflowing queries
        }
        // levels until one segment is left (segments of the first level are the
        // 2,048-centroid ranges, whether read from the table or the kept slots)
        const float *in_s = lvl0_s;
        const int32_t *in_id = lvl0_id;
        int64_t in_ld = lvl0_ld, M = L.table ? nlist : (int64_t)L.nseg * L.cap;
        const int *in_cnt = lvl0_cnt;
        int64_t M_left = nlist;
        int buf = 0;
        while (M_left > kSelectSeg) {
            launch_select(in_s, in_id, in_ld, n, M, nprobe, cand_id[buf], cand_s[buf], L.lvl, only,
                          in_cnt, st);
            in_s = cand_s[buf];
            in_id = cand_id[buf];
            in_ld = L.lvl;
            in_cnt = nullptr;
            M_left = level_entries(M_left, nprobe);
            M = M_left;
            buf ^= 1;
        }
        launch_select(in_s, in_id, in_ld, n, M, nprobe, o, cs, nprobe, only, in_cnt, st);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace sieve
