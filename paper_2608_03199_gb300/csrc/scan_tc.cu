// scan_tc.cu -- the grouped queries x partition-rows contraction on the
// tcgen05 tensor cores, with the fused tau / top-k / stop-line epilogue
// (the within-partition search of Sec. 4.1 and Sec. 5 for large groups).
//
// A tile is (partition p, up to 128 items of p's group).  Its 128 gathered
// queries form the MMA's M side; the partition's rows stream through in
// chunks of 256 (N); d is covered in K-blocks of 32 fp32 (one 128-byte
// swizzle row).  fp32 accuracy comes from an error-compensated split: every
// operand x is stored as hi = tf32(x) and lo = tf32(x - hi), and each K step
// issues three kind::tf32 MMAs, hi*hi + hi*lo + lo*hi, accumulated in fp32 in
// tensor memory.  The dropped lo*lo term and the rounding of lo are about
// 2^-22 of |q_i x_i| each, so a similarity is off by at most a few 1e-7 for
// unit vectors.
//
// Warp roles (416 threads, one block per SM, persistent over tiles):
//   warps 0-7   converters: load a stage (128 query half-rows + 256 row
//               K-blocks) from global memory, split hi/lo, store both in the
//               swizzled layout, arrive on the stage's "full" barrier
//   warp 8      allocates 512 tensor-memory columns (two 256-column
//               accumulators); lane 0 issues the MMAs and commits each stage
//               to its "empty" barrier and each finished chunk to "dfull"
//   warps 9-12  epilogue: thread i owns tensor-memory lane i = the tile's
//               i-th query; it reads its 256 scores of a chunk, keeps rows
//               with s >= tau (self excluded) in a private top-k, and after
//               the last chunk writes the item's local result and raises
//               the query's stop line on a hit
// Every mbarrier wait is bounded; a wait that gives up marks the block as
// aborted (SIEVE_ETIMEOUT in the status word), every role leaves its loop,
// outstanding MMAs are drained (bounded) and tensor memory is freed.
#include "search.cuh"
#include "tcgen05.cuh"

namespace sieve {

namespace {
constexpr int kM = 128;                  // queries per tile = tensor-memory lanes
constexpr int kN = 256;                  // partition rows per chunk = MMA N
constexpr int kKB = 32;                  // fp32 per K-block
constexpr int kConvWarps = 8;
constexpr int kMmaWarp = 8;
constexpr int kEpiWarp0 = 9;
constexpr int kTcThreads = 13 * 32;
constexpr uint32_t A_BYTES = kM * 128;   // one K-block of the tile's queries
constexpr uint32_t B_BYTES = kN * 128;   // one K-block of a row chunk
constexpr uint32_t STAGE_BYTES = 2 * A_BYTES + 2 * B_BYTES;   // hi and lo of both
constexpr int kStages = 2;
constexpr uint32_t kTmemCols = 2 * kN;
constexpr uint32_t kWaitPolls = 1u << 24;
constexpr uint32_t kIdesc = tc::idesc_tf32(kM, kN);
}  // namespace

size_t scan_tc_smem_bytes(int k) {
    return 1024 + (size_t)kStages * STAGE_BYTES + (size_t)kM * k * (sizeof(float) + sizeof(long long));
}

// store one K-block segment of a row as hi/lo tf32 pairs in the 128-byte
// swizzled layout: 16-byte chunk c of row r lives at chunk c ^ (r & 7)
template <int NCHUNK>
__device__ __forceinline__ void store_split(unsigned char *hi_tile, unsigned char *lo_tile, int row,
                                            int chunk0, const float4 (&v)[NCHUNK]) {
#pragma unroll
    for (int c = 0; c < NCHUNK; ++c) {
        const uint32_t off = (uint32_t)row * 128u + (uint32_t)(((chunk0 + c) ^ (row & 7)) << 4);
        uint4 h, l;
        h.x = tc::to_tf32(v[c].x);
        h.y = tc::to_tf32(v[c].y);
        h.z = tc::to_tf32(v[c].z);
        h.w = tc::to_tf32(v[c].w);
        l.x = tc::to_tf32(v[c].x - __uint_as_float(h.x));
        l.y = tc::to_tf32(v[c].y - __uint_as_float(h.y));
        l.z = tc::to_tf32(v[c].z - __uint_as_float(h.z));
        l.w = tc::to_tf32(v[c].w - __uint_as_float(h.w));
        *reinterpret_cast<uint4 *>(hi_tile + off) = h;
        *reinterpret_cast<uint4 *>(lo_tile + off) = l;
    }
}

__global__ void __launch_bounds__(kTcThreads, 1) k_scan_tc(SearchArgs a) {
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[kStages], empty_bar[kStages], dfull_bar[2],
        dempty_bar[2], drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int s_abort;

    unsigned char *base = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int k = a.k, d = a.d;
    float *kept_s = reinterpret_cast<float *>(base + kStages * STAGE_BYTES);
    long long *kept_id = reinterpret_cast<long long *>(kept_s + kM * k);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    Ctl *ctl = a.ctl;
    const int n_tiles = ctl->n_tc_tiles;
    const int nkb = (int)ceil_div(d, kKB);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&full_bar[s], kConvWarps * 32);
            tc::mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(&dfull_bar[b], 1);
            tc::mbar_init(&dempty_bar[b], 4 * 32);
        }
        tc::mbar_init(&drain_bar, 1);
        s_abort = 0;
        tc::mbar_init_fence();
    }
    if (warp == kMmaWarp) tc::tmem_alloc(&tmem_slot, kTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = tmem_slot;

    // bounded wait; gives up early once another role has aborted
    auto wait = [&](uint64_t *bar, uint32_t parity) -> bool {
        for (uint32_t it = 0; it < kWaitPolls; ++it) {
            if (tc::mbar_try_wait(bar, parity)) return true;
            if ((it & 255u) == 255u && *(volatile int *)&s_abort) return false;
        }
        atomicExch(&s_abort, 1);
        atomicExch(&ctl->status, SIEVE_ETIMEOUT);
        return false;
    };

    if (warp < kConvWarps) {
        // ---------------- converters ----------------
        const int pt = threadIdx.x;          // 0..255: B row of a chunk
        const int arow = pt >> 1, ahalf = pt & 1;
        uint32_t s = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
            const int4 tile = a.tc_tiles[t];
            const int p = tile.x, ib = tile.y, ni = tile.z;
            const int64_t r_begin = a.off[p];
            const int64_t np = a.off[p + 1] - r_begin;
            const int nch = (int)ceil_div(np, kN);
            const float *qrow = nullptr;
            if (arow < ni) qrow = a.Q + (int64_t)a.item_q[a.bucketed[ib + arow]] * d;
            for (int ch = 0; ch < nch; ++ch) {
                const int64_t brow = (int64_t)ch * kN + pt;
                const float *xrow = brow < np ? a.X + (r_begin + brow) * d : nullptr;
                for (int kb = 0; kb < nkb; ++kb, ++s) {
                    const uint32_t st = s & 1u, ph = (s >> 1) & 1u;
                    if (!wait(&empty_bar[st], ph ^ 1u)) goto conv_done;
                    unsigned char *stage = base + st * STAGE_BYTES;
                    {
                        float4 v[8];
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            const int col = kb * kKB + 4 * c;
                            v[c] = (xrow && col < d) ? __ldg(reinterpret_cast<const float4 *>(xrow + col))
                                                     : make_float4(0.f, 0.f, 0.f, 0.f);
                        }
                        store_split<8>(stage + 2 * A_BYTES, stage + 2 * A_BYTES + B_BYTES, pt, 0, v);
                    }
                    {
                        float4 u[4];
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const int col = kb * kKB + ahalf * 16 + 4 * c;
                            u[c] = (qrow && col < d) ? __ldg(reinterpret_cast<const float4 *>(qrow + col))
                                                     : make_float4(0.f, 0.f, 0.f, 0.f);
                        }
                        store_split<4>(stage, stage + A_BYTES, arow, ahalf * 4, u);
                    }
                    tc::fence_proxy_async_smem();
                    tc::mbar_arrive(&full_bar[st]);
                }
            }
        }
    conv_done:;
    } else if (warp == kMmaWarp) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            uint32_t s = 0, c = 0;
            bool ok = true;
            for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x) {
                const int4 tile = a.tc_tiles[t];
                const int64_t np = a.off[tile.x + 1] - a.off[tile.x];
                const int nch = (int)ceil_div(np, kN);
                for (int ch = 0; ok && ch < nch; ++ch, ++c) {
                    const uint32_t buf = c & 1u, dph = (c >> 1) & 1u;
                    if (!(ok = wait(&dempty_bar[buf], dph ^ 1u))) break;
                    tc::fence_after_sync();
                    const uint32_t dt = tmem + buf * kN;
                    for (int kb = 0; kb < nkb; ++kb, ++s) {
                        const uint32_t st = s & 1u, ph = (s >> 1) & 1u;
                        if (!(ok = wait(&full_bar[st], ph))) break;
                        tc::fence_after_sync();
                        const uint32_t sa = tc::smem_u32(base + st * STAGE_BYTES);
                        const uint32_t a_hi = sa, a_lo = sa + A_BYTES;
                        const uint32_t b_hi = sa + 2 * A_BYTES, b_lo = b_hi + B_BYTES;
#pragma unroll
                        for (int ks = 0; ks < kKB / 8; ++ks) {
                            const uint32_t o = ks * 32;
                            tc::mma_tf32(dt, tc::desc_k_sw128(a_lo + o), tc::desc_k_sw128(b_hi + o), kIdesc,
                                         (kb > 0 || ks > 0) ? 1u : 0u);
                            tc::mma_tf32(dt, tc::desc_k_sw128(a_hi + o), tc::desc_k_sw128(b_lo + o), kIdesc, 1u);
                            tc::mma_tf32(dt, tc::desc_k_sw128(a_hi + o), tc::desc_k_sw128(b_hi + o), kIdesc, 1u);
                        }
                        tc::mma_commit(&empty_bar[st]);
                    }
                    if (ok) tc::mma_commit(&dfull_bar[buf]);
                }
            }
            // every MMA issued by this thread has finished once drain_bar flips
            // (waited for even after an abort, within the poll limit)
            tc::mma_commit(&drain_bar);
            for (uint32_t it = 0; it < kWaitPolls; ++it)
                if (tc::mbar_try_wait(&drain_bar, 0u)) break;
        }
        __syncwarp();
    } else {
        // ---------------- epilogue ----------------
        const int quarter = warp & 3;        // tensor-memory lanes 32*quarter ..
        const int slot = quarter * 32 + lane;
        float *ks_ = kept_s + slot * k;
        long long *ki_ = kept_id + slot * k;
        const float tau = a.tau;
        uint32_t c = 0;
        bool ok = true;
        for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x) {
            const int4 tile = a.tc_tiles[t];
            const int p = tile.x, ib = tile.y, ni = tile.z;
            const int64_t r_begin = a.off[p];
            const int64_t np = a.off[p + 1] - r_begin;
            const int nch = (int)ceil_div(np, kN);
            const bool valid = slot < ni;
            int item = 0, q = 0, rank = 0;
            long long qid = (long long)-0x7fffffffffffffffll - 1;
            if (valid) {
                item = a.bucketed[ib + slot];
                q = a.item_q[item];
                rank = a.item_rank[item];
                if (a.qids) qid = a.qids[q];
            }
            int kn = 0;
            for (int ch = 0; ch < nch; ++ch, ++c) {
                const uint32_t buf = c & 1u, dph = (c >> 1) & 1u;
                ok = __all_sync(0xffffffffu, wait(&dfull_bar[buf], dph));
                if (!ok) break;
                tc::fence_after_sync();
#pragma unroll 1
                for (int cc = 0; cc < kN / 32; ++cc) {
                    float v[32];
                    tc::tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + buf * kN + cc * 32, v);
                    if (valid) {
                        const int64_t col0 = (int64_t)ch * kN + cc * 32;
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            if (v[j] >= tau && col0 + j < np) {
                                const long long id = a.ids[r_begin + col0 + j];
                                if (id == qid) continue;
                                const float sc = v[j];
                                if (kn == k && !ranks_before(sc, id, ks_[k - 1], ki_[k - 1])) continue;
                                int i = kn < k ? kn++ : k - 1;
                                while (i > 0 && ranks_before(sc, id, ks_[i - 1], ki_[i - 1])) {
                                    ks_[i] = ks_[i - 1];
                                    ki_[i] = ki_[i - 1];
                                    --i;
                                }
                                ks_[i] = sc;
                                ki_[i] = id;
                            }
                        }
                    }
                }
                tc::fence_before_sync();
                tc::mbar_arrive(&dempty_bar[buf]);
            }
            if (!ok) break;
            if (valid) {
                for (int j = 0; j < kn; ++j) {
                    a.res_s[(int64_t)item * k + j] = ks_[j];
                    a.res_id[(int64_t)item * k + j] = ki_[j];
                }
                a.res_cnt[item] = kn;
                if (kn > 0) {   // a hit at rank j commits ranks up to min(j + W, nprobe)
                    const long long reach = (long long)rank + a.W;
                    atomicMax(&a.S[q], reach < a.nprobe ? (int)reach : a.nprobe);
                }
            }
            if (slot == 0) {
                atomicAdd(&ctl->tot_rows, (unsigned long long)np);
                atomicAdd(&ctl->tot_pairs, (unsigned long long)np * (unsigned long long)ni);
                atomicAdd(&ctl->tot_rows_tc, (unsigned long long)np);
                atomicAdd(&ctl->tot_pairs_tc, (unsigned long long)np * (unsigned long long)ni);
            }
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

cudaError_t prepare_scan_tc(int k) {
    return cudaFuncSetAttribute(k_scan_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)scan_tc_smem_bytes(k));
}

void enqueue_scan_tc(const SearchArgs &a, cudaStream_t st) {
    k_scan_tc<<<num_sms(), kTcThreads, scan_tc_smem_bytes(a.k), st>>>(a);
}

}  // namespace sieve
