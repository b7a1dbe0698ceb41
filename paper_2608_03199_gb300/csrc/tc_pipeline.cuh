// tc_pipeline.cuh -- a persistent tcgen05 contraction pipeline shared by the
// grouped scan and the centroid ranking: S = A * B^T for tiles of 128 rows
// of A (queries) against all rows of a B range (partition rows or
// centroids), in fp32 accuracy through a 3xTF32 split, handed chunk by chunk
// to a per-row epilogue.
//
// A tile's 128 A rows form the MMA's M side; B streams through in chunks of
// Mode::kN rows (the MMA N); d is covered in K-blocks of 32 fp32 (one
// 128-byte swizzle row).  Every operand x is stored as hi = tf32(x) and
// lo = tf32(x - hi); each K step issues three kind::tf32 MMAs,
// lo*hi + hi*lo + hi*hi, accumulated in fp32 in tensor memory.  The dropped
// lo*lo term and the rounding of lo are about 2^-22 of |a_i b_i| each, so a
// unit-vector similarity is off by at most a few 1e-7.
//
// Warp roles (416 threads, one block per SM):
//   warps 0-7   converters: load a stage (128 A half-rows and one K-block of
//               the B chunk) from global memory, split hi/lo, store both in
//               the swizzled layout, arrive on the stage's "full" barrier
//   warp 8      allocates 2 * kN tensor-memory columns (two accumulators);
//               lane 0 issues the MMAs, commits each stage to its "empty"
//               barrier and each finished chunk to "dfull"
//   warps 9-12  epilogue: thread i owns tensor-memory lane i = A row i of the
//               tile; it reads that row's kN scores of a chunk (Mode::Epi),
//               then releases the accumulator ("dempty")
// Every mbarrier wait is bounded: a wait that gives up marks the block as
// aborted (SIEVE_ETIMEOUT in the mode's status word), every role leaves its
// loop, the issued MMAs are drained (bounded) and tensor memory is freed.
#pragma once

#include "search.cuh"
#include "tcgen05.cuh"

namespace sieve {
namespace tcp {

constexpr int kM = 128;                  // A rows per tile = tensor-memory lanes
constexpr int kKB = 32;                  // fp32 per K-block
constexpr int kConvWarps = 8;
constexpr int kMmaWarp = 8;
constexpr int kThreads = 13 * 32;
constexpr int kStages = 2;
constexpr uint32_t kWaitPolls = 1u << 24;
constexpr uint32_t A_BYTES = kM * 128;   // one K-block of the tile's A rows

template <int N>
struct Geometry {
    static constexpr uint32_t B_BYTES = N * 128;
    static constexpr uint32_t STAGE_BYTES = 2 * A_BYTES + 2 * B_BYTES;   // hi + lo of A and B
    static constexpr uint32_t TMEM_COLS = 2 * N;
    static constexpr size_t smem_bytes(size_t epi_bytes) {
        return 1024 + (size_t)kStages * STAGE_BYTES + epi_bytes;
    }
};

// store NCHUNK 16-byte chunks of a row, starting at logical chunk chunk0, as
// hi/lo tf32 pairs in the 128-byte swizzled layout (chunk c of row r sits
// at chunk c ^ (r & 7))
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

template <int NCHUNK>
__device__ __forceinline__ void load_chunks(const float *row, int col0, int d, float4 (&v)[NCHUNK]) {
#pragma unroll
    for (int c = 0; c < NCHUNK; ++c) {
        const int col = col0 + 4 * c;
        v[c] = (row && col < d) ? __ldg(reinterpret_cast<const float4 *>(row + col))
                                : make_float4(0.f, 0.f, 0.f, 0.f);
    }
}

// Mode provides: kN; Args; Tile; num_tiles(a); tile(a, t) with fields
// ni (A rows used) and nb (B rows); a_row(a, T, i) / b_row(a, T, r) (row
// pointers or nullptr past the end); status(a); d(a); epi_bytes(a); and the
// per-thread epilogue Epi with begin(a, T, slot, smem), chunk(a, T, col0,
// v[32], ncol), end(a, T).
template <class Mode>
__device__ __forceinline__ void run_pipeline(const typename Mode::Args &a, unsigned char *smem_raw) {
    constexpr int kN = Mode::kN;
    using G = Geometry<kN>;
    constexpr uint32_t kIdesc = tc::idesc_tf32(kM, kN);
    constexpr int kBThreadsPerRow = (kConvWarps * 32) / kN;   // 1 (N = 256) or 2 (N = 128)
    constexpr int kBChunks = 8 / kBThreadsPerRow;
    static_assert(kBThreadsPerRow * kN == kConvWarps * 32, "one or two converters per B row");

    __shared__ __align__(8) uint64_t full_bar[kStages], empty_bar[kStages], dfull_bar[2],
        dempty_bar[2], drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int s_abort;

    unsigned char *base = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    unsigned char *epi_smem = base + kStages * G::STAGE_BYTES;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tiles = Mode::num_tiles(a);
    const int d = Mode::d(a);
    const int nkb = (int)ceil_div(d, kKB);
    int *status = Mode::status(a);

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
    if (warp == kMmaWarp) tc::tmem_alloc(&tmem_slot, G::TMEM_COLS);
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
        atomicExch(status, SIEVE_ETIMEOUT);
        return false;
    };

    if (warp < kConvWarps) {
        // ---------------- converters ----------------
        const int pt = threadIdx.x;
        const int arow = pt >> 1, ahalf = pt & 1;
        const int brow_l = pt / kBThreadsPerRow, bpart = pt % kBThreadsPerRow;
        uint32_t s = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
            const typename Mode::Tile T = Mode::tile(a, t);
            const int nch = (int)ceil_div(T.nb, kN);
            const float *arow_p = Mode::a_row(a, T, arow);
            for (int ch = 0; ch < nch; ++ch) {
                const float *brow_p = Mode::b_row(a, T, (int64_t)ch * kN + brow_l);
                for (int kb = 0; kb < nkb; ++kb, ++s) {
                    const uint32_t st = s & 1u, ph = (s >> 1) & 1u;
                    if (!wait(&empty_bar[st], ph ^ 1u)) goto conv_done;
                    unsigned char *stage = base + st * G::STAGE_BYTES;
                    {
                        float4 v[kBChunks];
                        load_chunks<kBChunks>(brow_p, kb * kKB + bpart * kBChunks * 4, d, v);
                        store_split<kBChunks>(stage + 2 * A_BYTES, stage + 2 * A_BYTES + G::B_BYTES,
                                              brow_l, bpart * kBChunks, v);
                    }
                    {
                        float4 u[4];
                        load_chunks<4>(arow_p, kb * kKB + ahalf * 16, d, u);
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
                const typename Mode::Tile T = Mode::tile(a, t);
                const int nch = (int)ceil_div(T.nb, kN);
                for (int ch = 0; ok && ch < nch; ++ch, ++c) {
                    const uint32_t buf = c & 1u, dph = (c >> 1) & 1u;
                    if (!(ok = wait(&dempty_bar[buf], dph ^ 1u))) break;
                    tc::fence_after_sync();
                    const uint32_t dt = tmem + buf * kN;
                    for (int kb = 0; kb < nkb; ++kb, ++s) {
                        const uint32_t st = s & 1u, ph = (s >> 1) & 1u;
                        if (!(ok = wait(&full_bar[st], ph))) break;
                        tc::fence_after_sync();
                        const uint32_t sa = tc::smem_u32(base + st * G::STAGE_BYTES);
                        const uint32_t a_hi = sa, a_lo = sa + A_BYTES;
                        const uint32_t b_hi = sa + 2 * A_BYTES, b_lo = b_hi + G::B_BYTES;
#pragma unroll
                        for (int ks = 0; ks < kKB / 8; ++ks) {
                            const uint32_t o = ks * 32;
                            tc::mma_tf32(dt, tc::desc_k_sw128(a_lo + o), tc::desc_k_sw128(b_hi + o),
                                         kIdesc, (kb > 0 || ks > 0) ? 1u : 0u);
                            tc::mma_tf32(dt, tc::desc_k_sw128(a_hi + o), tc::desc_k_sw128(b_lo + o),
                                         kIdesc, 1u);
                            tc::mma_tf32(dt, tc::desc_k_sw128(a_hi + o), tc::desc_k_sw128(b_hi + o),
                                         kIdesc, 1u);
                        }
                        tc::mma_commit(&empty_bar[st]);
                    }
                    if (ok) tc::mma_commit(&dfull_bar[buf]);
                }
            }
            // every MMA issued by this thread has finished once drain_bar
            // flips (waited for even after an abort, within the poll limit)
            tc::mma_commit(&drain_bar);
            for (uint32_t it = 0; it < kWaitPolls; ++it)
                if (tc::mbar_try_wait(&drain_bar, 0u)) break;
        }
        __syncwarp();
    } else {
        // ---------------- epilogue ----------------
        const int quarter = warp & 3;        // tensor-memory lanes 32 * quarter ..
        const int slot = quarter * 32 + lane;
        uint32_t c = 0;
        bool ok = true;
        typename Mode::Epi epi;
        for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x) {
            const typename Mode::Tile T = Mode::tile(a, t);
            const int nch = (int)ceil_div(T.nb, kN);
            epi.begin(a, T, slot, epi_smem);
            for (int ch = 0; ch < nch; ++ch, ++c) {
                const uint32_t buf = c & 1u, dph = (c >> 1) & 1u;
                ok = __all_sync(0xffffffffu, wait(&dfull_bar[buf], dph));
                if (!ok) break;
                tc::fence_after_sync();
#pragma unroll 1
                for (int cc = 0; cc < kN / 32; ++cc) {
                    float v[32];
                    tc::tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + buf * kN + cc * 32, v);
                    const int64_t col0 = (int64_t)ch * kN + cc * 32;
                    const int64_t left = T.nb - col0;
                    epi.chunk(a, T, col0, v, left < 32 ? (int)left : 32);
                }
                tc::fence_before_sync();
                tc::mbar_arrive(&dempty_bar[buf]);
            }
            if (!ok) break;
            epi.end(a, T);
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, G::TMEM_COLS);
    }
}

}  // namespace tcp
}  // namespace sieve
