// tc_bulk.cuh -- the tensor-core contraction fed from the tensor-core layout
// (tc_layout.cu): S = A * B^T for tiles of 128 A rows (queries) against every
// block of 128 B rows (a partition's rows, or the centroids), with the scaled
// fp16 split of tc_pipeline.cuh and the same per-row epilogues.
//
// The B operand arrives pre-split, in tile byte order: a block's K-blocks (32 KB
// each: hi then lo) are contiguous, and one bulk copy lands two of them as a
// stage in shared memory, a few stages deep, with no thread touching the bytes.
// B operands that are exact in fp16 (codes) have no lo part: 16 KB per K-block.  The tile's 128 A rows are
// split once per tile straight into tensor memory (lane i = A row i, two fp16
// per 32-bit column, hi and lo of each K-block side by side), so shared memory
// holds nothing but B stages and the epilogue's lists.
//
// Tensor memory (512 columns): two 128-column fp32 accumulators (three when
// d <= 128), then the tile's A: 64 columns per K-block of 64 elements (32 hi,
// 32 lo); d <= 256.  K steps of 16 that lie wholly in the zero padding of the
// last K-block are not issued (d = 96: six of eight).
// A screening mode (one product per K step, hi halves only) copies just the
// hi half of each K-block of B and keeps only A's hi columns (32 per
// K-block), so three accumulators fit.
//
// Warp roles (448 threads, one block per SM):
//   warps 0-7   A writers: warp w writes lanes 32 (w % 4) .. +31 for the
//               K-blocks kb with kb % 2 == w / 4.  For each tile they load
//               their query row early (an L2 prefetch of the whole row, then
//               the K-block's values into registers), and only then wait until
//               the previous tile's last MMAs on that K-block are done
//               ("a_empty[kb]"), split the values, store them with tcgen05.st
//               and publish the K-block ("a_full[kb]")
//   warp 8      lane 0 takes the block's next tile (an atomic work counter,
//               or a static stride when the mode has none) and hands it to the
//               other roles through a small ring in shared memory; it then
//               issues the tile's bulk copies of B stages ("b_full" with the
//               transfer byte count; waits on "b_empty")
//   warp 9      allocates the tensor memory; lane 0 issues the mode's one to
//               three kind::f16 MMAs per K step (A from tensor memory, B from
//               shared memory)
//   warps 10-13 epilogue: thread i owns tensor-memory lane i = A row i; it
//               hands its row of a chunk (scores x 2^16) to Mode::Epi
//
// Two sub-tiles (a mode with kSub = 2): a tile is 256 A rows, two sets of 128
// in tensor memory side by side, and every B stage feeds the MMAs of both, so
// each byte of B streamed into shared memory does twice the work.  Where the
// A rows are few per tile and many B chunks follow (the centroid ranking),
// writing A is rare and the epilogue is the busy role: warps 0-3 write A
// (every K-block of both sub-tiles), warp 4 is the producer, warp 5 the MMA
// issuer and warps 6-13 the epilogue, 6-9 on sub-tile 0 and 10-13 on
// sub-tile 1 (warp w reads tensor-memory lanes 32 (w % 4) .. +31).  Each
// sub-tile has its own accumulator, handed to its epilogue as soon as its
// MMAs of the chunk are issued, so one sub-tile's epilogue runs while the
// other's MMAs do.
// Every wait is bounded; giving up sets SIEVE_ETIMEOUT in the mode's status
// word, all roles leave their loops, the issued MMAs and copies are drained
// (bounded) and tensor memory is freed.
#pragma once

#include <cuda_fp16.h>

#include "search.cuh"
#include "tc_pipeline.cuh"
#include "tcgen05.cuh"

namespace sieve {
namespace tcb {

constexpr int kN = 128;                       // B rows per chunk = MMA N = tensor-layout block
constexpr int kAWriterWarps = 8;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kThreads = 14 * 32;
constexpr int kMaxKb = 4;                     // A in tensor memory: d <= 256
constexpr int kMaxStages = 8;                 // barrier slots for B stages
constexpr int kStagesMax = 5;                 // stages beyond five did not time faster
constexpr uint32_t kKbBytes = 32768;          // one K-block of 128 rows: hi 16 KB + lo 16 KB
constexpr uint32_t kTmemCols = 512;
constexpr int kMaxAcc = 3;                    // accumulator slots (barriers)
constexpr uint32_t kWaitPolls = 1u << 24;
constexpr int kRing = 8;                      // tiles handed from the scheduler to the other roles
constexpr uint32_t kRingReaders = kAWriterWarps + 1 + 4;   // A-writer warps, MMA lane, epilogue warps

constexpr uint32_t kKbBytesHi = 16384;        // one K-block of 128 rows with no lo part (codes)
constexpr int kKbPerStage = 2;                // two K-blocks per B stage: one copy and one
                                              // commit per 24 (or 16) MMAs; timed 8-10%
                                              // faster than one K-block per stage
constexpr uint32_t kStageBytes = kKbPerStage * kKbBytes;       // 64 KB
constexpr uint32_t kStageBytesHi = kKbPerStage * kKbBytesHi;   // 32 KB

// shared memory: 1 KB alignment slack, the B stages, the epilogue's bytes
__host__ __device__ inline size_t smem_bytes(int stages, size_t epi_bytes,
                                             uint32_t stage_bytes = kStageBytes) {
    return 1024 + (size_t)stages * stage_bytes + epi_bytes;
}

// B stages that fit beside the epilogue (0 when the pipeline does not apply)
inline int stages_for(int nkb, size_t epi_bytes, size_t smem_limit, uint32_t stage_bytes = kStageBytes,
                      int max_stages = kStagesMax) {
    if (nkb > kMaxKb) return 0;
    const size_t base = smem_bytes(0, epi_bytes, stage_bytes);
    if (smem_limit < base) return 0;
    int s = (int)((smem_limit - base) / stage_bytes);
    if (s > max_stages) s = max_stages;
    if (s > kMaxStages) s = kMaxStages;
    return s >= 2 ? s : 0;
}

// Modes whose B operand has a lo part (a split fp32 value: three products
// per K step) and modes whose B is exact in fp16 (integer codes: B = hi only,
// two products, half the stage)
template <class Mode, class = void>
struct b_has_lo { static constexpr bool value = true; };
template <class Mode>
struct b_has_lo<Mode, decltype((void)Mode::kBHasLo)> { static constexpr bool value = Mode::kBHasLo; };

// products per K step: 3 (lo_a hi_b + hi_a lo_b + hi_a hi_b), 2 (B exact in
// fp16: lo_a b + hi_a b) or 1 (a screen: hi_a hi_b, the hi halves of a split
// B copied alone)
template <class Mode, class = void>
struct mma_products { static constexpr int value = b_has_lo<Mode>::value ? 3 : 2; };
template <class Mode>
struct mma_products<Mode, decltype((void)Mode::kProducts)> { static constexpr int value = Mode::kProducts; };

// B rows per chunk (the MMA's N): Mode::kNB if given, else 128 (one block of
// the tensor layout).  192 is for a screen of two sub-tiles at d <= 128: its
// A (2 x 64 columns) and two 192-column accumulators fill tensor memory, and
// each MMA instruction covers half as many columns again -- the issuing
// thread, not the tensor pipe, bounds such a screen.  A 192-row chunk spans
// two layout blocks: rows 0-127 or 64-127 of one and the start of the next.
template <class Mode, class = void>
struct chunk_rows { static constexpr int value = kN; };
template <class Mode>
struct chunk_rows<Mode, decltype((void)Mode::kNB)> { static constexpr int value = Mode::kNB; };

// sub-tiles of 128 A rows per tile: Mode::kSub if given (1 or 2), else 1
template <class Mode, class = void>
struct sub_tiles { static constexpr int value = 1; };
template <class Mode>
struct sub_tiles<Mode, decltype((void)Mode::kSub)> { static constexpr int value = Mode::kSub; };

// tensor-memory columns of one sub-tile's A: 64 per K-block (hi and lo), 32
// for a screen (hi alone)
__host__ __device__ constexpr uint32_t a_cols(int nkb, int products) {
    return (uint32_t)nkb * (products == 1 ? 32u : 64u);
}

// 128-column accumulators beside A: one sub-tile takes three when its A
// takes at most 128 columns, else two; two sub-tiles take two, accumulator j
// always sub-tile j's, so that each accumulator's barriers have one reader
// group and phases cannot be skipped
__host__ __device__ constexpr uint32_t acc_slots(int nkb, int products, int sub) {
    return sub == 1 ? ((products == 1 || nkb <= 2) ? 3u : 2u) : 2u;
}

// whether a pipeline of sub sub-tiles fits tensor memory at this d
__host__ __device__ constexpr bool sub_fits(int nkb, int products, int sub) {
    return nkb <= kMaxKb && (uint32_t)sub * a_cols(nkb, products) + 2u * kN <= kTmemCols;
}

// polls of the epilogue's accumulator wait: the mode's epi_wait_polls(a) if
// it has one (a testing aid that lets that wait give up early; 0 = default),
// else kWaitPolls.  No other wait takes it: every drain keeps the full limit.
template <class Mode, class = void>
struct has_epi_wait { static constexpr bool value = false; };
template <class Mode>
struct has_epi_wait<Mode, decltype((void)Mode::epi_wait_polls(*(const typename Mode::Args *)nullptr))> {
    static constexpr bool value = true;
};
template <class Mode>
__device__ __forceinline__ uint32_t epi_wait_polls(const typename Mode::Args &a) {
    if constexpr (has_epi_wait<Mode>::value) {
        const uint32_t n = Mode::epi_wait_polls(a);
        return n ? n : kWaitPolls;
    } else {
        return kWaitPolls;
    }
}

// one 32-column group of an accumulator row to the mode's epilogue
template <class Epi, class Args, class Tile>
__device__ __forceinline__ void hand(Epi &epi, const Args &a, const Tile &T, int64_t col0,
                                     const uint32_t (&r)[32]) {
    float v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
    const int64_t left = T.nb - col0;
    epi.chunk(a, T, col0, v, left < 32 ? (int)left : 32);
}

// The MMAs of one B stage for one sub-tile, fully unrolled: K1 K steps of 16
// in the stage's first K-block and K2 in its second (0: none).  a0 = the
// sub-tile's A columns of that first K-block (hi; lo 32 columns on), b0 = the
// shared-memory descriptor of the stage's first K-block; a K step moves A by
// 8 columns and B's start address by 32 bytes (2 in the descriptor's 16-byte
// units; shared addresses stay below the field's 2^14 limit, so no carry).
// acc_first: whether the first MMA accumulates (0 at a chunk's first K step).
// One straight run of MMAs with their operands a constant off two bases: the
// single issuing thread keeps up with the tensor pipe.
template <int kProd, int K1, int K2, uint32_t kKbStageBytes>
__device__ __forceinline__ void issue_stage(uint32_t dt, uint32_t a0, uint64_t b0, uint32_t acc_first,
                                            uint32_t idesc) {
    constexpr uint32_t kAKbT = kProd == 1 ? 32 : 64;                       // A columns per K-block
    constexpr uint64_t kKbDesc = kKbStageBytes >> 4;                         // B K-block in 16-byte units
    constexpr uint64_t kLoDesc = (kKbBytes / 2) >> 4;                        // hi to lo of a split K-block
#pragma unroll
    for (int j = 0; j < K1 + K2; ++j) {
        const int kb = j < K1 ? 0 : 1, ks = j < K1 ? j : j - K1;
        const uint32_t a = a0 + (uint32_t)kb * kAKbT + (uint32_t)ks * 8u;
        const uint64_t bh = b0 + (uint64_t)kb * kKbDesc + 2u * (uint64_t)ks;
        const uint32_t acc = j == 0 ? acc_first : 1u;
        if constexpr (kProd == 3) {        // lo_a hi_b + hi_a lo_b + hi_a hi_b
            tc::mma_f16_ta(dt, a + 32u, bh, idesc, acc);
            tc::mma_f16_ta(dt, a, bh + kLoDesc, idesc, 1u);
            tc::mma_f16_ta(dt, a, bh, idesc, 1u);
        } else if constexpr (kProd == 2) { // B exact in fp16: lo_a b + hi_a b
            tc::mma_f16_ta(dt, a + 32u, bh, idesc, acc);
            tc::mma_f16_ta(dt, a, bh, idesc, 1u);
        } else {                           // a screen: hi_a hi_b
            tc::mma_f16_ta(dt, a, bh, idesc, acc);
        }
    }
}

// issue_stage for a run-time K-step pattern: a stage's first K-block has k1
// steps (1..4) and its second k2 (0..4, only after a full first block)
template <int kProd, uint32_t kKbStageBytes>
__device__ __forceinline__ void issue_stage_rt(int k1, int k2, uint32_t dt, uint32_t a0, uint64_t b0,
                                               uint32_t acc_first, uint32_t idesc) {
    constexpr uint32_t B = kKbStageBytes;
    switch (k1 * 8 + k2) {
        case 4 * 8 + 4: issue_stage<kProd, 4, 4, B>(dt, a0, b0, acc_first, idesc); break;
        case 4 * 8 + 3: issue_stage<kProd, 4, 3, B>(dt, a0, b0, acc_first, idesc); break;
        case 4 * 8 + 2: issue_stage<kProd, 4, 2, B>(dt, a0, b0, acc_first, idesc); break;
        case 4 * 8 + 1: issue_stage<kProd, 4, 1, B>(dt, a0, b0, acc_first, idesc); break;
        case 4 * 8 + 0: issue_stage<kProd, 4, 0, B>(dt, a0, b0, acc_first, idesc); break;
        case 3 * 8 + 0: issue_stage<kProd, 3, 0, B>(dt, a0, b0, acc_first, idesc); break;
        case 2 * 8 + 0: issue_stage<kProd, 2, 0, B>(dt, a0, b0, acc_first, idesc); break;
        default: issue_stage<kProd, 1, 0, B>(dt, a0, b0, acc_first, idesc); break;
    }
}

// Mode provides (in addition to what tc_pipeline.cuh asks): Epi::prefetch(a,
// T, ch) and Epi::start(a, T, ch), called by every epilogue lane of a warp
// before and after the wait for chunk ch's accumulator; b_block(a, T, ch)
// = pointer to the tensor-layout bytes of the tile's ch-th block of B rows;
// tile_counter(a) = a zeroed global int the blocks draw tiles from (nullptr:
// block b takes tiles b, b + gridDim.x, ...).
template <class Mode>
__device__ __forceinline__ void run_bulk(const typename Mode::Args &a, unsigned char *smem_raw,
                                         int stages) {
    constexpr int kNB = chunk_rows<Mode>::value;               // B rows per chunk = MMA N
    constexpr uint32_t kIdesc = tc::idesc_f16(tcp::kM, kNB);
    constexpr int kProd = mma_products<Mode>::value;
    constexpr bool kLo = kProd == 3;                          // B's lo half in the stage
    // bytes of one K-block of B in a stage (kNB rows)
    constexpr uint32_t kKbB = (kLo ? kKbBytes : kKbBytesHi) / kN * kNB;
    // bytes of one K-block of B in global memory: a screen copies the hi half
    // of each K-block of the split layout, one copy per K-block
    constexpr uint32_t kSrcKb = b_has_lo<Mode>::value ? kKbBytes : kKbBytesHi;
    // A's tensor-memory columns per K-block: hi and lo (64), or a screen's hi
    // half alone (32)
    constexpr uint32_t kAKb = kProd == 1 ? 32 : 64;
    constexpr int kKs = kKbPerStage;                          // K-blocks per B stage
    constexpr uint32_t kStage = kKs * kKbB;                    // bytes of one B stage
    constexpr int kSub = sub_tiles<Mode>::value;
    static_assert(kSub == 1 || kSub == 2, "one or two sub-tiles");
    static_assert(kNB == kN || (kNB == 192 && kProd == 1 && kSub == 2 && kSrcKb == kKbBytes),
                  "192-row chunks: a screen of two sub-tiles over the split layout");
    // warp roles: A writers, producer, MMA issuer, epilogue (4 warps per sub-tile)
    constexpr int kAW = kSub == 1 ? kAWriterWarps : 4;
    constexpr int kAWGroups = kAW / 4;                         // K-block classes of A writers
    constexpr int kProdW = kAW, kMmaW = kAW + 1, kEpiW0 = kAW + 2;
    static_assert(kEpiW0 + 4 * kSub == kThreads / 32, "every warp has a role");
    static_assert(kAW + 1 + 4 * kSub == (int)kRingReaders, "ring readers");
    __shared__ __align__(8) uint64_t a_full[kMaxKb], a_empty[kMaxKb], b_full[kMaxStages],
        b_empty[kMaxStages], dfull_bar[kMaxAcc], dempty_bar[kMaxAcc], drain_bar, ring_full[kRing],
        ring_empty[kRing];
    __shared__ int ring_tile[kRing];
    __shared__ uint32_t tmem_slot;
    __shared__ int s_abort;

    unsigned char *base = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tiles = Mode::num_tiles(a);
    const int d = Mode::d(a);
    const int nkb = (int)ceil_div(d, 64);
    int *status = Mode::status(a);
    // a d whose A does not fit tensor memory (the host never launches one):
    // report it and leave before any barrier or tensor memory is set up
    if (!sub_fits(nkb, kProd, kSub) ||
        (uint32_t)kSub * a_cols(nkb, kProd) + 2u * (uint32_t)kNB > kTmemCols) {
        if (threadIdx.x == 0) atomicExch(status, SIEVE_EINVAL);
        return;
    }
    const uint32_t nacc = acc_slots(nkb, kProd, kSub);
    const uint32_t aTile = a_cols(nkb, kProd);                 // A columns of one sub-tile
    unsigned char *Bst = base;                                 // stages x kStage
    unsigned char *epi_smem = Bst + (size_t)stages * kStage;
    int *tile_counter = Mode::tile_counter(a);

    if (threadIdx.x == 0) {
        for (int kb = 0; kb < kMaxKb; ++kb) {
            tc::mbar_init(&a_full[kb], 4 * 32);
            tc::mbar_init(&a_empty[kb], 1);
        }
        for (int s = 0; s < kMaxStages; ++s) {
            tc::mbar_init(&b_full[s], 1);
            tc::mbar_init(&b_empty[s], 1);
        }
        for (uint32_t b = 0; b < (uint32_t)kMaxAcc; ++b) {
            tc::mbar_init(&dfull_bar[b], 1);
            tc::mbar_init(&dempty_bar[b], 4 * 32);
        }
        for (int r = 0; r < kRing; ++r) {
            tc::mbar_init(&ring_full[r], 1);
            tc::mbar_init(&ring_empty[r], kRingReaders);
        }
        tc::mbar_init(&drain_bar, 1);
        s_abort = 0;
        tc::mbar_init_fence();
    }
    if (warp == kMmaW) tc::tmem_alloc(&tmem_slot, kTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = tmem_slot;
    const uint32_t tA = tmem + nacc * kNB;                     // A after the accumulators

    auto wait_n = [&](uint64_t *bar, uint32_t parity, uint32_t polls) -> bool {
        // a phase that has completed already is seen by a non-blocking test:
        // a (blocking) try_wait costs about 200 cycles of the waiting thread
        // even then, which the single MMA-issuing thread cannot afford
        if (tc::mbar_test_wait(bar, parity)) return true;
        // a shortened limit polls without blocking (try_wait may suspend the
        // thread for a hardware-chosen time, which would stretch the limit)
        const bool quick = polls < kWaitPolls;
        for (uint32_t it = 0; it < polls; ++it) {
            if (quick ? tc::mbar_test_wait(bar, parity) : tc::mbar_try_wait(bar, parity)) return true;
            if ((it & 255u) == 255u && *(volatile int *)&s_abort) return false;
        }
        atomicExch(&s_abort, 1);
        atomicExch(status, SIEVE_ETIMEOUT);
        return false;
    };
    auto wait = [&](uint64_t *bar, uint32_t parity) -> bool { return wait_n(bar, parity, kWaitPolls); };
    const uint32_t epi_wait = epi_wait_polls<Mode>(a);
    // the i-th tile of this block from the ring, read by a whole warp (one
    // arrival per warp); false when the wait gave up.  t < 0 ends the loop.
    auto ring_take_warp = [&](uint32_t i, int &t) -> bool {
        const uint32_t slot = i % kRing, ph = (i / kRing) & 1u;
        if (!__all_sync(0xffffffffu, wait(&ring_full[slot], ph))) return false;
        t = *(volatile int *)&ring_tile[slot];
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&ring_empty[slot]);
        return true;
    };

    if (warp < kAW) {
        // ---------------- A writers ----------------
        const int quarter = warp & 3, group = warp >> 2;
        const int row = quarter * 32 + lane;
        const uint32_t lane_bits = (uint32_t)(quarter * 32) << 16;
        uint32_t u = 0;
        bool ok = true;
        for (uint32_t i = 0; ok; ++i) {
            int t;
            if (!ring_take_warp(i, t) || t < 0) break;
            const typename Mode::Tile T = Mode::tile(a, t);
            if (T.nb <= 0) continue;
            if (group == 0)
                for (int h = 0; h < kSub; ++h) {
                    const float *rp = Mode::a_row(a, T, row + h * tcp::kM);
                    if (rp) tc::prefetch_l2(rp, (uint32_t)d * 4u);   // d % 4 == 0
                }
            for (int kb = group; ok && kb < nkb; kb += kAWGroups) {
#pragma unroll 1
                for (int h = 0; h < kSub; ++h) {
                    const float *rp = Mode::a_row(a, T, row + h * tcp::kM);
                    float4 x[16];
#pragma unroll
                    for (int q4 = 0; q4 < 16; ++q4) x[q4] = tcp::load_f4(rp, kb * 64 + 4 * q4, d);
                    if (h == 0) {
                        if (!(ok = __all_sync(0xffffffffu, wait(&a_empty[kb], (u & 1u) ^ 1u)))) break;
                        tc::fence_after_sync();
                    }
#pragma unroll
                    for (int half = 0; half < 2; ++half) {     // 32 elements = 16 columns per half
                        uint32_t hi[16], lo[16];
#pragma unroll
                        for (int q4 = 0; q4 < 8; ++q4) {
                            const float4 v = x[half * 8 + q4];
                            tcp::split2(v.x, v.y, hi[2 * q4], lo[2 * q4]);
                            tcp::split2(v.z, v.w, hi[2 * q4 + 1], lo[2 * q4 + 1]);
                        }
                        const uint32_t col = tA + (uint32_t)h * aTile + (uint32_t)kb * kAKb + (uint32_t)half * 16;
                        tc::tmem_st16(col + lane_bits, hi);
                        if constexpr (kProd > 1) tc::tmem_st16(col + 32 + lane_bits, lo);
                    }
                }
                if (!ok) break;
                tc::tmem_st_wait();
                tc::fence_before_sync();
                tc::mbar_arrive(&a_full[kb]);
            }
            ++u;
        }
    } else if (warp == kProdW) {
        // ---------------- tile scheduler + B producer ----------------
        if (lane == 0) {
            uint32_t s = 0;
            // the block's i-th tile into ring slot i % kRing (t < 0: no more)
            auto publish = [&](uint32_t i, int &t) -> bool {
                const uint32_t slot = i % kRing, ph = (i / kRing) & 1u;
                if (!wait(&ring_empty[slot], ph ^ 1u)) return false;
                t = tile_counter ? atomicAdd(tile_counter, 1) : (int)(blockIdx.x + i * gridDim.x);
                if (t >= n_tiles) t = -1;
                ring_tile[slot] = t;
                tc::mbar_arrive(&ring_full[slot]);   // release: the tile id is visible with the phase
                return true;
            };
            int cur = -1;
            bool ok = publish(0, cur);
            for (uint32_t i = 0; ok && cur >= 0; ++i) {
                // the next tile is published before this one's copies are
                // issued: the A writers gather its rows while this tile's MMAs
                // run, instead of after its last copy
                int nxt = -1;
                if (!(ok = publish(i + 1, nxt))) break;
                const typename Mode::Tile T = Mode::tile(a, cur);
                cur = nxt;
                const int nch = (int)ceil_div(T.nb, kNB);
                const int nblk = (int)ceil_div(T.nb, kN);             // layout blocks of the tile's B
                for (int ch = 0; ok && ch < nch; ++ch) {
                    if constexpr (kNB != kN) {
                        // a 192-row chunk: rows r0 .. r0 + 191 of the tile's B, from
                        // block r0 / 128 (from its row r0 % 128) and the next block
                        // (while it exists: rows past the tile's blocks are not
                        // copied, and their columns are never read); the hi half of
                        // each K-block, rows at 128 bytes, lands at the chunk row
                        const int r0 = ch * kNB, b0 = r0 / kN, o0 = r0 % kN;
                        const uint32_t n0 = (uint32_t)(kN - o0);
                        const uint32_t n1 = b0 + 1 < nblk ? (uint32_t)kNB - n0 : 0u;
                        const unsigned char *p0 = Mode::b_block(a, T, b0);
                        const unsigned char *p1 = n1 ? Mode::b_block(a, T, b0 + 1) : nullptr;
                        for (int kb = 0; kb < nkb; kb += kKs) {
                            const uint32_t st = s % stages, sph = (s / stages) & 1u;
                            const int nk = nkb - kb < kKs ? nkb - kb : kKs;
                            if (!(ok = wait(&b_empty[st], sph ^ 1u))) break;
                            tc::mbar_arrive_expect_tx(&b_full[st], (uint32_t)nk * (n0 + n1) * 128u);
                            for (int j = 0; j < nk; ++j) {
                                unsigned char *dst = Bst + (size_t)st * kStage + (size_t)j * kKbB;
                                tc::bulk_g2s(dst, p0 + (size_t)(kb + j) * kSrcKb + (size_t)o0 * 128u, n0 * 128u,
                                             &b_full[st]);
                                if (n1)
                                    tc::bulk_g2s(dst + (size_t)n0 * 128u, p1 + (size_t)(kb + j) * kSrcKb, n1 * 128u,
                                                 &b_full[st]);
                            }
                            ++s;
                        }
                        continue;
                    }
                    // a block's K-blocks are contiguous: a stage is one copy
                    const unsigned char *src = Mode::b_block(a, T, ch);
                    for (int kb = 0; kb < nkb; kb += kKs) {
                        const uint32_t st = s % stages, sph = (s / stages) & 1u;
                        const uint32_t bytes = (uint32_t)(nkb - kb < kKs ? nkb - kb : kKs) * kKbB;
                        if (!(ok = wait(&b_empty[st], sph ^ 1u))) break;
                        tc::mbar_arrive_expect_tx(&b_full[st], bytes);
                        if constexpr (kSrcKb == kKbB) {
                            tc::bulk_g2s(Bst + (size_t)st * kStage, src + (size_t)kb * kKbB, bytes,
                                         &b_full[st]);
                        } else {   // the hi halves of this stage's K-blocks
                            for (uint32_t j = 0; j * kKbB < bytes; ++j)
                                tc::bulk_g2s(Bst + (size_t)st * kStage + j * kKbB,
                                             src + ((size_t)kb + j) * kSrcKb, kKbB, &b_full[st]);
                        }
                        ++s;
                    }
                }
            }
            // no copy may still be landing when the block exits: wait (bounded)
            // for the last copy issued into each stage
            for (uint32_t j = s > (uint32_t)stages ? s - stages : 0; j < s; ++j)
                for (uint32_t it = 0; it < kWaitPolls; ++it)
                    if (tc::mbar_try_wait(&b_full[j % stages], (j / stages) & 1u)) break;
        }
        __syncwarp();
    } else if (warp == kMmaW) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            uint32_t s = 0, c = 0, u = 0;   // c: accumulator uses, kSub per chunk
            bool ok = true;
            // the descriptor of stage 0's first K-block; stage st is st * kStage
            // bytes on (the start-address field does not carry: shared
            // addresses stay below 2^18)
            const uint64_t b_desc0 = tc::desc_k_sw128(tc::smem_u32(Bst));
            for (uint32_t i = 0; ok; ++i) {
                const uint32_t slot = i % kRing, rph = (i / kRing) & 1u;
                if (!(ok = wait(&ring_full[slot], rph))) break;
                const int t = *(volatile int *)&ring_tile[slot];
                tc::mbar_arrive(&ring_empty[slot]);
                if (t < 0) break;
                const typename Mode::Tile T = Mode::tile(a, t);
                const int nch = (int)ceil_div(T.nb, kNB);
                if (nch == 0) continue;
                for (int ch = 0; ok && ch < nch; ++ch, c += kSub) {
                    if constexpr (kSub == 1) {   // the chunk's accumulator
                        if (!(ok = wait(&dempty_bar[c % nacc], ((c / nacc) & 1u) ^ 1u))) break;
                        tc::fence_after_sync();
                    }
                    for (int kb0 = 0; kb0 < nkb; kb0 += kKs, ++s) {
                        const uint32_t st = s % stages, ph = (s / stages) & 1u;
                        const int kb1 = nkb - kb0 < kKs ? nkb : kb0 + kKs;   // this stage's K-blocks
                        const bool last = kb1 == nkb;                       // the chunk's last stage
                        if (ch == 0)
                            for (int kb = kb0; ok && kb < kb1; ++kb) ok = wait(&a_full[kb], u & 1u);
                        if (!ok || !(ok = wait(&b_full[st], ph))) break;
                        tc::fence_after_sync();
                        // K steps of 16 that hold any of the d elements (the rest of
                        // the last K-block is zero padding), per K-block of the stage
                        const int k1 = d - kb0 * 64 >= 64 ? 4 : (d - kb0 * 64 + 15) / 16;
                        const int k2 = kb1 - kb0 < 2 ? 0 : d - (kb0 + 1) * 64 >= 64 ? 4 : (d - (kb0 + 1) * 64 + 15) / 16;
                        const uint64_t b_stage = b_desc0 + (uint64_t)st * (kStage >> 4);
#pragma unroll 1
                        for (int h = 0; ok && h < kSub; ++h) {
                            if (kSub > 1 && kb0 == 0) {   // sub-tile h's accumulator, just before its MMAs
                                if (!(ok = wait(&dempty_bar[(c + h) % nacc], (((c + h) / nacc) & 1u) ^ 1u))) break;
                                tc::fence_after_sync();
                            }
                            const uint32_t dt = tmem + ((c + h) % nacc) * kNB;
                            issue_stage_rt<kProd, kKbB>(k1, k2, dt, tA + (uint32_t)h * aTile + (uint32_t)kb0 * kAKb,
                                                        b_stage, kb0 > 0 ? 1u : 0u, kIdesc);
                            // with two sub-tiles, the first sub-tile's accumulator is
                            // handed over before the second's MMAs are issued
                            if (kSub > 1 && last && h + 1 < kSub) tc::mma_commit(&dfull_bar[(c + h) % nacc]);
                        }
                        if (!ok) break;
                        tc::mma_commit(&b_empty[st]);
                        // the tile's last reads of these K-blocks of A: they may be
                        // overwritten by the next tile once they are done
                        if (ch == nch - 1)
                            for (int kb = kb0; kb < kb1; ++kb) tc::mma_commit(&a_empty[kb]);
                    }
                    if (ok) tc::mma_commit(&dfull_bar[(c + kSub - 1) % nacc]);
                }
                ++u;
            }
            tc::mma_commit(&drain_bar);
            for (uint32_t it = 0; it < kWaitPolls; ++it)
                if (tc::mbar_try_wait(&drain_bar, 0u)) break;
        }
        __syncwarp();
    } else {
        // ---------------- epilogue ----------------
        const int quarter = warp & 3;                      // the lanes this warp may read
        const int h = (warp - kEpiW0) >> 2;                // its sub-tile
        const int slot = h * tcp::kM + quarter * 32 + lane;
        uint32_t c = h;
        bool ok = true;
        typename Mode::Epi epi;
        for (uint32_t i = 0; ok; ++i) {
            int t;
            if (!ring_take_warp(i, t) || t < 0) break;
            const typename Mode::Tile T = Mode::tile(a, t);
            const int nch = (int)ceil_div(T.nb, kNB);
            epi.begin(a, T, slot, epi_smem);
            for (int ch = 0; ch < nch; ++ch, c += kSub) {
                const uint32_t buf = c % nacc, dph = (c / nacc) & 1u;
                epi.prefetch(a, T, ch);   // per-chunk loads, in flight during the wait
                ok = __all_sync(0xffffffffu, wait_n(&dfull_bar[buf], dph, epi_wait));
                if (!ok) break;
                epi.start(a, T, ch);
                tc::fence_after_sync();
                // pairs of 32-column loads, each pair in flight together; the
                // accumulator is released as soon as the last pair has landed,
                // before its columns are handed to the mode
                const uint32_t taddr = tmem + ((uint32_t)(quarter * 32) << 16) + buf * kNB;
                const int64_t col0 = (int64_t)ch * kNB;
                uint32_t ra[32], rb[32];
#pragma unroll
                for (int pr = 0; pr < kNB / 64; ++pr) {
                    tc::tmem_ld32_issue(taddr + pr * 64, ra);
                    tc::tmem_ld32_issue(taddr + pr * 64 + 32, rb);
                    tc::tmem_ld_wait(ra);
                    tc::tmem_ld_wait(rb);
                    if (pr == kNB / 64 - 1) {
                        tc::fence_before_sync();
                        tc::mbar_arrive(&dempty_bar[buf]);
                    }
                    hand(epi, a, T, col0 + pr * 64, ra);
                    hand(epi, a, T, col0 + pr * 64 + 32, rb);
                }
            }
            if (!ok) break;
            epi.end(a, T);
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == kMmaW) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace tcb
}  // namespace sieve
