// rank_tc.cu -- centroid ranking on the tcgen05 tensor cores (Sec. 2.3,
// Sec. 4.1: P_i = the nprobe centroids with the largest inner product with
// q_i, best first, equal scores by lower centroid id), for nlist <= 2048.
//
// Two kernels per chunk of queries:
//   k_rank_tc  the 3xTF32 pipeline of tc_pipeline.cuh: 128 consecutive
//              queries (A rows) against all centroids (B rows, 128 per
//              chunk); each epilogue thread stores its query's scores into a
//              score table [queries][ld] in the caller's workspace
//   k_select   one warp per query: the query's scores sit in registers
//              (nlist / 32 per lane); the exact nprobe-th largest score is
//              found bit by bit (32 rounds of "how many scores are >= t"),
//              the entries above it plus the lowest-id entries equal to it
//              are gathered, and a warp bitonic network sorts them by
//              (score desc, id asc).
#include "tc_bulk.cuh"
#include "tc_pipeline.cuh"

namespace sieve {

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
};

__device__ int g_rank_status_sink;

struct RankMode {
    using Args = RankArgs;
    static constexpr int kN = 128;
    struct Tile {
        int64_t q0;
        int ni;
        int64_t nb;
    };
    __device__ static int num_tiles(const Args &a) { return (int)ceil_div(a.nq, tcp::kM); }
    // every tile costs the same: a static stride over the blocks
    __device__ static int *tile_counter(const Args &) { return nullptr; }
    __device__ static int d(const Args &a) { return a.d; }
    __device__ static int *status(const Args &a) { return a.status ? a.status : &g_rank_status_sink; }
    __device__ static Tile tile(const Args &a, int t) {
        Tile T;
        T.q0 = (int64_t)t * tcp::kM;
        T.ni = (int)(a.nq - T.q0 < tcp::kM ? a.nq - T.q0 : tcp::kM);
        T.nb = a.nlist;
        return T;
    }
    __device__ static const float *a_row(const Args &a, const Tile &T, int i) {
        return i < T.ni ? a.Q + (T.q0 + i) * a.d : nullptr;
    }
    __device__ static const float *b_row(const Args &a, const Tile &T, int64_t r) {
        return r < T.nb ? a.C + r * a.d : nullptr;
    }
    __device__ static const unsigned char *b_block(const Args &a, const Tile &, int ch) {
        return a.tc_cent + (int64_t)ch * ((a.d + 63) / 64) * kTcBlockBytes;
    }
    struct Epi {
        float *row;
        __device__ void begin(const Args &a, const Tile &T, int slot, unsigned char *) {
            row = slot < T.ni ? a.scores + (T.q0 + slot) * a.ld : nullptr;
        }
        // v holds the chunk's raw accumulator values: scores x 2^16
        __device__ void chunk(const Args &a, const Tile &, int64_t col0, const float (&v)[32], int ncol) {
            if (!row || ncol <= 0) return;   // ld is a multiple of 32: whole 32-column groups fit
            constexpr float kS = 1.f / 65536.f;
            float4 *dst = reinterpret_cast<float4 *>(row + col0);
#pragma unroll
            for (int j = 0; j < 8; ++j)
                dst[j] = make_float4(v[4 * j] * kS, v[4 * j + 1] * kS, v[4 * j + 2] * kS, v[4 * j + 3] * kS);
        }
        __device__ void end(const Args &, const Tile &) {}
        __device__ void stage(const Args &, const Tile &, int64_t, int) {}
        __device__ void use_staged(int) {}
    };
    static constexpr bool kStage = false;
};

__global__ void __launch_bounds__(tcp::kThreads, 1) k_rank_tc(RankArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcp::run_pipeline<RankMode>(a, smem_raw);
}

int rank_bulk_stages(int d) { return tcb::stages_for((int)ceil_div(d, 64), 0, 232448 - 128); }

__global__ void __launch_bounds__(tcb::kThreads, 1) k_rank_bulk(RankArgs a, int stages) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RankMode>(a, smem_raw, stages);
}

// ---------------------------------------------------------------------------
// selection: monotone map of fp32 to uint32 (larger float -> larger key); -0
// is mapped as +0 so that equal scores have equal keys
__device__ __forceinline__ uint32_t order_key(float s) {
    const uint32_t u = __float_as_uint(s + 0.f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

constexpr int kSelectWarps = 4;
constexpr int kSelectMaxR = 4;   // lane order statistics used for the lower bracket

__device__ __forceinline__ int warp_sum(int x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

template <int KPL>
__device__ __forceinline__ int count_ge(const uint32_t (&key)[KPL], uint32_t t) {
    int c = 0;
#pragma unroll
    for (int j = 0; j < KPL; ++j) c += key[j] >= t;
    return warp_sum(c);
}

// One warp per query.  T* = the nprobe-th largest key.  The search keeps a
// threshold T <= T* with C = #{keys >= T} >= nprobe and refines T bit by bit
// (the largest T with at least nprobe keys >= T) until C fits the sort
// buffer; it starts from the common high bits of a bracket L <= T* <= U
// (U = the largest key; L = the smallest over lanes of each lane's
// ceil(nprobe / 32)-th largest key, so at least nprobe keys are >= L).  The
// C candidates >= T contain the nprobe best, which a bitonic sort by
// (score desc, id asc) puts first.  When C never fits (many equal scores),
// the search ends at T = T* and takes the keys > T* plus the lowest-id keys
// equal to it.  P: a power of two >= nprobe; the buffer holds 2P entries.
template <int KPL>   // scores per lane: nlist <= 32 * KPL
__global__ void __launch_bounds__(kSelectWarps * 32) k_select(const float *__restrict__ scores,
                                                              int64_t ld, int64_t nq, int nlist,
                                                              int nprobe, int P,
                                                              int32_t *__restrict__ order,
                                                              float *__restrict__ cscores) {
    extern __shared__ __align__(16) unsigned char sel_smem[];
    const int cap = 2 * P;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *bs = reinterpret_cast<float *>(sel_smem) + warp * 2 * cap;   // cap scores, then cap ids
    int *bc = reinterpret_cast<int *>(bs + cap);
    const int64_t q = (int64_t)blockIdx.x * kSelectWarps + warp;
    if (q >= nq) return;
    const float *row = scores + q * ld;
    float s[KPL];
    uint32_t key[KPL];
#pragma unroll
    for (int j = 0; j < KPL; ++j) {
        const int c = j * 32 + lane;
        s[j] = c < nlist ? row[c] : 0.f;
        key[j] = c < nlist ? order_key(s[j]) : 0u;   // padding ranks below every score
    }
    // bracket: per lane the r largest keys (a small insertion network)
    const int r = (nprobe + 31) / 32;
    uint32_t m[kSelectMaxR] = {0u, 0u, 0u, 0u};
    if (r <= 2) {
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            m[1] = max(m[1], min(m[0], key[j]));
            m[0] = max(m[0], key[j]);
        }
    } else {
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
    }
    uint32_t U = m[0];
    uint32_t L = r == 1 ? m[0] : r == 2 ? m[1] : r == 3 ? m[2] : r == 4 ? m[3] : 0u;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        U = max(U, __shfl_xor_sync(0xffffffffu, U, o));
        L = min(L, __shfl_xor_sync(0xffffffffu, L, o));
    }
    int b;
    uint32_t T;
    if (L == U) {
        b = -1;
        T = L;
    } else {
        b = 31 - __clz(L ^ U);                                // highest bit where they differ
        T = b == 31 ? 0u : (L & ~((2u << b) - 1u));           // their common high bits
    }
    int C = count_ge(key, T);
    for (; b >= 0 && C > cap; --b) {
        const uint32_t t = T | (1u << b);
        const int cnt = count_ge(key, t);
        if (cnt >= nprobe) {
            T = t;
            C = cnt;
        }
    }
    const unsigned below = (1u << lane) - 1u;
    int pos = 0;
    if (C <= cap) {
        // every key >= T, in increasing id order (id = 32 j + lane)
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            const bool sel = key[j] >= T && j * 32 + lane < nlist;
            const unsigned sb = __ballot_sync(0xffffffffu, sel);
            if (sel) {
                const int p = pos + __popc(sb & below);
                bs[p] = s[j];
                bc[p] = j * 32 + lane;
            }
            pos += __popc(sb);
        }
    } else {
        // T == T*: the keys above it, then the lowest-id keys equal to it
        int gt = 0;
#pragma unroll
        for (int j = 0; j < KPL; ++j) gt += key[j] > T;
        const int ties_wanted = nprobe - warp_sum(gt);   // >= 1
        int ties_seen = 0;
#pragma unroll
        for (int j = 0; j < KPL; ++j) {
            const bool tie = key[j] == T && j * 32 + lane < nlist;
            const unsigned tb = __ballot_sync(0xffffffffu, tie);
            const bool sel = key[j] > T || (tie && ties_seen + __popc(tb & below) < ties_wanted);
            const unsigned sb = __ballot_sync(0xffffffffu, sel);
            if (sel) {
                const int p = pos + __popc(sb & below);
                bs[p] = s[j];
                bc[p] = j * 32 + lane;
            }
            pos += __popc(sb);
            ties_seen += __popc(tb);
        }
    }
    int S = 1;   // sort size: a power of two >= pos (pos <= cap)
    while (S < pos) S <<= 1;
    for (int p = pos + lane; p < S; p += 32) {
        bs[p] = -__int_as_float(0x7f800000);
        bc[p] = INT32_MAX;
    }
    __syncwarp();
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
    for (int p = lane; p < nprobe; p += 32) {
        order[q * nprobe + p] = bc[p];
        if (cscores) cscores[q * nprobe + p] = bs[p];
    }
}

// ---------------------------------------------------------------------------
bool rank_tc_supported(int64_t nlist, int nprobe) { return nlist <= kRankTcMaxNlist && nprobe <= nlist; }

int64_t rank_tc_ld(int64_t nlist) { return round_up(nlist, 32); }

int64_t rank_tc_chunk(int64_t nq, int64_t nlist) {
    const int64_t per_q = rank_tc_ld(nlist) * (int64_t)sizeof(float);
    int64_t c = kRankScratchBytes / per_q;
    c = c / tcp::kM * tcp::kM;
    if (c < tcp::kM) c = tcp::kM;
    return nq < c ? nq : c;
}

size_t rank_tc_scratch_bytes(int64_t nq, int64_t nlist) {
    return (size_t)(rank_tc_chunk(nq, nlist) * rank_tc_ld(nlist) * (int64_t)sizeof(float));
}

static size_t tc_smem() { return tcp::Geometry<RankMode::kN>::smem_bytes(0); }

static int pow2_at_least(int x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

template <int KPL>
static cudaError_t set_select_attr(int P) {
    return cudaFuncSetAttribute(k_select<KPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kSelectWarps * 2 * (2 * P) * 4);
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
    return e;
}

cudaError_t enqueue_rank_tc(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                            int nprobe, int32_t *order, float *cscores, float *scratch, int *status,
                            cudaStream_t st, const unsigned char *tc_cent) {
    const int bulk_stages = tc_cent ? rank_bulk_stages(d) : 0;
    const int64_t ld = rank_tc_ld(nlist);
    const int64_t chunk = rank_tc_chunk(nq, nlist);
    const int P = pow2_at_least(nprobe);
    const int kpl = pow2_at_least((int)ceil_div(nlist, 32));
    for (int64_t q0 = 0; q0 < nq; q0 += chunk) {
        const int64_t n = nq - q0 < chunk ? nq - q0 : chunk;
        RankArgs a{Q + q0 * d, n, C, nlist, d, scratch, ld, status, tc_cent};
        const int tiles = (int)ceil_div(n, tcp::kM);
        if (bulk_stages)
            k_rank_bulk<<<std::min(tiles, num_sms()), tcb::kThreads,
                          tcb::smem_bytes(bulk_stages, 0), st>>>(a, bulk_stages);
        else
            k_rank_tc<<<std::min(tiles, num_sms()), tcp::kThreads, tc_smem(), st>>>(a);
        const unsigned blocks = (unsigned)ceil_div(n, kSelectWarps);
        const size_t smem = (size_t)kSelectWarps * 2 * (2 * P) * 4;
        int32_t *o = order + q0 * nprobe;
        float *cs = cscores ? cscores + q0 * nprobe : nullptr;
        switch (kpl) {
            case 1: k_select<1><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
            case 2: k_select<2><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
            case 4: k_select<4><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
            case 8: k_select<8><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
            case 16: k_select<16><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
            case 32: k_select<32><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
            default: k_select<64><<<blocks, kSelectWarps * 32, smem, st>>>(scratch, ld, n, (int)nlist, nprobe, P, o, cs); break;
        }
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace sieve
