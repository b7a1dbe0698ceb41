// tc_pipeline.cuh -- a persistent tcgen05 contraction pipeline shared by the
// grouped scan and the centroid ranking: S = A * B^T for tiles of 128 rows
// of A (queries) against all rows of a B range (partition rows or
// centroids), to fp32 accuracy through an error-compensated fp16 split,
// handed chunk by chunk to a per-row epilogue.
//
// A tile's 128 A rows form the MMA's M side; B streams through in chunks of
// Mode::kN rows (the MMA N); d is covered in K-blocks of 64 elements (one
// 128-byte swizzle row of fp16).  Every operand x is scaled by 2^8 and stored
// as hi = fp16(256 x) and lo = fp16(256 x - hi); each K step issues three
// kind::f16 MMAs, lo*hi + hi*lo + hi*hi, accumulated in fp32 in tensor
// memory, and the epilogue multiplies by 2^-16 (exact).  For |x| <= 1,
// |256 x - hi| <= 2^-12 |256 x|, the rounding of lo adds 2^-11 of that, and
// the dropped lo*lo term is 2^-24 of |256 a 256 b|: a unit-vector similarity
// is off by a few 1e-7 at most, as with a 3xTF32 split, at half the shared
// memory bytes per product (the scale keeps lo out of fp16's subnormal range
// whenever |x| >= 2^-11; below that its absolute error is under 2^-33).
//
// Warp roles (672 threads, one block per SM):
//   warps 0-15  converters: load one K-block of the tile's 128 A rows and of
//               the current B chunk from global memory (before waiting for
//               the stage to free up), split hi/lo, store both in the
//               swizzled layout, arrive on the stage's "full" barrier
//   warp 16     allocates 2 * kN tensor-memory columns (two accumulators);
//               lane 0 issues the MMAs, commits each stage to its "empty"
//               barrier and each finished chunk to "dfull"
//   warps 17-20 epilogue: thread i owns tensor-memory lane i = A row i of the
//               tile; it hands that row's kN raw accumulator values of a chunk
//               (scores x 2^16) to Mode::Epi, then releases the accumulator
//               ("dempty")
// Every mbarrier wait is bounded: a wait that gives up marks the block as
// aborted (SIEVE_ETIMEOUT in the mode's status word), every role leaves its
// loop, the issued MMAs are drained (bounded) and tensor memory is freed.
#pragma once

#include <cuda_fp16.h>

#include "search.cuh"
#include "tcgen05.cuh"

namespace sieve {
namespace tcp {

constexpr int kM = 128;                  // A rows per tile = tensor-memory lanes
constexpr int kKB = 64;                  // elements per K-block (128 bytes of fp16)
constexpr int kConvWarps = 16;
constexpr int kConvThreads = kConvWarps * 32;
constexpr int kMmaWarp = 16;
constexpr float kSplitScale = 256.f;               // operands scaled by 2^8 ...
constexpr float kUnscale = 1.f / 65536.f;          // ... products by 2^16
constexpr int kThreads = 21 * 32;
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

// A converter thread handles one float4 (4 consecutive elements) of a row at
// a time: it becomes 8 bytes of fp16 in the hi tile and 8 in the lo tile, one
// half of a 16-byte chunk.  Chunk c of row r sits at chunk c ^ (r & 7) (the
// 128-byte swizzle the descriptors name).  Sixteen consecutive threads cover
// one row's K-block, so a warp reads two rows' 256 contiguous bytes each.
__device__ __forceinline__ float4 load_f4(const float *row, int col, int d) {
    return (row && col < d) ? __ldg(reinterpret_cast<const float4 *>(row + col))
                            : make_float4(0.f, 0.f, 0.f, 0.f);
}

__device__ __forceinline__ void split2(float a, float b, uint32_t &hi, uint32_t &lo) {
    const float2 f = make_float2(a * kSplitScale, b * kSplitScale);
    const __half2 h = __float22half2_rn(f);
    const float2 back = __half22float2(h);
    const __half2 l = __float22half2_rn(make_float2(f.x - back.x, f.y - back.y));
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

// f = index of the float4 within the row's K-block (0..15)
__device__ __forceinline__ void store_f4(unsigned char *hi_tile, unsigned char *lo_tile, int row,
                                         int f, const float4 &x) {
    const uint32_t off =
        (uint32_t)row * 128u + (uint32_t)((((f >> 1) ^ (row & 7)) << 4) | ((f & 1) << 3));
    uint2 h, l;
    split2(x.x, x.y, h.x, l.x);
    split2(x.z, x.w, h.y, l.y);
    *reinterpret_cast<uint2 *>(hi_tile + off) = h;
    *reinterpret_cast<uint2 *>(lo_tile + off) = l;
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
    constexpr uint32_t kIdesc = tc::idesc_f16(kM, kN);
    constexpr int kRowsPerPass = kConvThreads / 16;      // 32 rows per pass of all converters
    constexpr int kAPasses = kM / kRowsPerPass;          // 4
    constexpr int kBPasses = kN / kRowsPerPass;          // 8 (N = 256) or 4 (N = 128)
    static_assert(kAPasses * kRowsPerPass == kM && kBPasses * kRowsPerPass == kN, "");

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
            tc::mbar_init(&full_bar[s], kConvThreads);
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
        // a completed phase is seen by a non-blocking test (a blocking
        // try_wait costs about 200 cycles even then)
        if (tc::mbar_test_wait(bar, parity)) return true;
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
        const int f = threadIdx.x & 15;          // float4 of the K-block
        const int r0 = threadIdx.x >> 4;         // first row; rows r0 + 32 i
        uint32_t s = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
            const typename Mode::Tile T = Mode::tile(a, t);
            const int nch = (int)ceil_div(T.nb, kN);
            const float *arow_p[kAPasses];
#pragma unroll
            for (int i = 0; i < kAPasses; ++i) arow_p[i] = Mode::a_row(a, T, r0 + kRowsPerPass * i);
            for (int ch = 0; ch < nch; ++ch) {
                for (int kb = 0; kb < nkb; ++kb, ++s) {
                    const uint32_t st = s & 1u, ph = (s >> 1) & 1u;
                    const int col = kb * kKB + 4 * f;
                    float4 bx[kBPasses], ax[kAPasses];
#pragma unroll
                    for (int i = 0; i < kBPasses; ++i)
                        bx[i] = load_f4(Mode::b_row(a, T, (int64_t)ch * kN + r0 + kRowsPerPass * i), col, d);
#pragma unroll
                    for (int i = 0; i < kAPasses; ++i) ax[i] = load_f4(arow_p[i], col, d);
                    if (!wait(&empty_bar[st], ph ^ 1u)) goto conv_done;
                    unsigned char *stage = base + st * G::STAGE_BYTES;
#pragma unroll
                    for (int i = 0; i < kBPasses; ++i)
                        store_f4(stage + 2 * A_BYTES, stage + 2 * A_BYTES + G::B_BYTES,
                                 r0 + kRowsPerPass * i, f, bx[i]);
#pragma unroll
                    for (int i = 0; i < kAPasses; ++i)
                        store_f4(stage, stage + A_BYTES, r0 + kRowsPerPass * i, f, ax[i]);
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
                        // K steps holding any of the d elements (the rest is zero padding)
                        const int kst = d - kb * kKB >= kKB ? kKB / 16 : (d - kb * kKB + 15) / 16;
#pragma unroll
                        for (int ks = 0; ks < kKB / 16; ++ks) {   // K = 16 fp16 = 32 bytes per MMA
                            if (ks >= kst) break;
                            const uint32_t o = ks * 32;
                            tc::mma_f16(dt, tc::desc_k_sw128(a_lo + o), tc::desc_k_sw128(b_hi + o),
                                        kIdesc, (kb > 0 || ks > 0) ? 1u : 0u);
                            tc::mma_f16(dt, tc::desc_k_sw128(a_hi + o), tc::desc_k_sw128(b_lo + o),
                                        kIdesc, 1u);
                            tc::mma_f16(dt, tc::desc_k_sw128(a_hi + o), tc::desc_k_sw128(b_hi + o),
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
