// scan_tc.cu -- the grouped queries x partition-rows contraction on the
// tcgen05 tensor cores with the fused tau / top-k / stop-line epilogue (the
// within-partition search of Sec. 4.1 and Sec. 5, for large groups).
//
// A tile is (partition p, up to 128 items of p's group): the items' queries
// are the A rows, p's rows are the B rows, streamed in chunks through the
// fp16-split pipelines (tc_bulk.cuh, tc_pipeline.cuh).  Epilogue thread i (the tile's i-th
// item) keeps the rows with s >= tau, other than the query itself, in a
// private top-k in shared memory; after p's last chunk it writes the item's
// local result and, on a hit at rank j, raises the query's stop line to
// min(j + W, nprobe) (Sec. 4.3).
#include "tc_bulk.cuh"
#include "tc_pipeline.cuh"

namespace sieve {

__device__ __forceinline__ int tc_nkb_dev(int d) { return (d + 63) / 64; }

// epilogue shared memory beyond the kept lists (bulk pipeline): per epilogue
// warp one 512-byte copy of a chunk's factors (the scan over codes) and two
// 1 KB buffers of row ids
constexpr size_t kEpiFacBytes = 4 * 512;
constexpr size_t kEpiIdsBytes = 4 * 2 * 1024;

// kRQ = false: exact inner products (B = the rows' hi / lo split);
// kRQ = true: RaBitQ-style estimates from the code layout (B = u - mid).
// kScreen (exact only): one product of the hi halves per pair screens every
// row, and the rows that may reach the threshold are scored again exactly
template <bool kRQ, bool kScreen = false>
struct ScanModeT {
    using Args = SearchArgs;
    static constexpr int kN = 256;
    static constexpr bool kBHasLo = !kRQ;
    static constexpr int kProducts = kScreen ? 1 : (kRQ ? 2 : 3);
    struct Tile {
        int p, ib, ni;
        int64_t r_begin, nb;
        int64_t blk0;       // p's first block in the bulk layout (codes for kRQ)
        const float *fac;   // kRQ: the factors x 2^-8 of p's rows (block order)
    };
    __device__ static int num_tiles(const Args &a) { return a.ctl->n_tc_tiles; }
    // tiles differ in cost (partition sizes are skewed): blocks draw them dynamically
    __device__ static int *tile_counter(const Args &a) { return &a.ctl->tc_tile_next; }
    __device__ static int d(const Args &a) { return a.d; }
    __device__ static int *status(const Args &a) { return &a.ctl->status; }
    __device__ static uint32_t epi_wait_polls(const Args &a) { return (uint32_t)a.wait_limit; }
    __device__ static Tile tile(const Args &a, int t) {
        const int4 x = a.tc_tiles[t];
        Tile T;
        T.p = x.x;
        T.ib = x.y;
        T.ni = x.z;
        T.r_begin = a.off[T.p];
        T.nb = a.off[T.p + 1] - T.r_begin;
        T.blk0 = kRQ ? a.rq_row_blocks[T.p] : (a.tc_row_blocks ? a.tc_row_blocks[T.p] : 0);
        T.fac = kRQ ? a.rq_fac + T.blk0 * kTcRows : nullptr;
        return T;
    }
    __device__ static const float *a_row(const Args &a, const Tile &T, int i) {
        const float *Qa = kRQ ? a.Qrot : a.Q;
        return i < T.ni ? Qa + (int64_t)a.item_q[a.bucketed[T.ib + i]] * a.d : nullptr;
    }
    __device__ static const float *b_row(const Args &a, const Tile &T, int64_t r) {
        return r < T.nb ? a.X + (T.r_begin + r) * a.d : nullptr;
    }
    __device__ static const unsigned char *b_block(const Args &a, const Tile &T, int ch) {
        if (kRQ) return a.rq_rows + (T.blk0 + ch) * (int64_t)tc_nkb_dev(a.d) * tcb::kKbBytesHi;
        return a.tc_rows + (T.blk0 + ch) * (int64_t)tc_nkb_dev(a.d) * kTcBlockBytes;
    }

    struct Epi {
        float *ks;
        long long *ki;
        int kn, item, q, rank, slot;
        float qc;   // kRQ: <q, c_p>, the centroid score of the item's rank
        float *fs;  // kRQ: this warp's copy of the chunk's 128 factors (shared memory)
        // kScreen: |q| of the item's query, the error-bound coefficients, the
        // largest row norm of each of the tile's 128-row blocks and that of
        // the current chunk (loaded before its accumulator wait)
        float qn, m_rel, m_abs, xn, xn_next;
        const float *bn;
        // bulk pipeline: this warp's two buffers of 128 row ids, filled by
        // asynchronous copies one chunk ahead; buffer ids_ch % 2 holds the
        // current chunk's (ids_ch < 0 on the converter pipeline, which reads
        // ids from global memory)
        long long *ids_b;
        int ids_ch;
        bool valid;
        long long qid;
        // the kept list is unordered while the tile runs; once it holds k
        // entries, (wst_s, wst_id) at wst_pos is the one that ranks last
        float wst_s;
        long long wst_id;
        int wst_pos;
        // entry j of thread slot's list sits at [j * kM + slot] (bank-conflict free)
        __device__ float &KS(int j) const { return ks[j * tcp::kM]; }
        __device__ long long &KI(int j) const { return ki[j * tcp::kM]; }
        __device__ void begin(const Args &a, const Tile &T, int slot_, unsigned char *smem) {
            slot = slot_;
            ks = reinterpret_cast<float *>(smem) + slot;
            ki = reinterpret_cast<long long *>(reinterpret_cast<float *>(smem) + tcp::kM * a.k) + slot;
            kn = 0;
            wst_s = 0.f;
            wst_id = 0;
            wst_pos = 0;
            valid = slot < T.ni;
            item = q = rank = 0;
            qid = (long long)-0x7fffffffffffffffll - 1;
            qc = 0.f;
            fs = reinterpret_cast<float *>(smem + (size_t)tcp::kM * a.k * 12) + (slot >> 5) * 128;
            ids_b = reinterpret_cast<long long *>(smem + (size_t)tcp::kM * a.k * 12 + kEpiFacBytes) +
                    (slot >> 5) * 2 * tcb::kN;
            ids_ch = -1;
            if (valid) {
                item = a.bucketed[T.ib + slot];
                q = a.item_q[item];
                rank = a.item_rank[item];
                if (a.qids) qid = a.qids[q];
                if (kRQ) qc = a.cscores[(int64_t)q * a.nprobe + rank - 1];
            }
            if constexpr (kScreen) {
                // the block norms follow the layout's blocks
                const int nkb = tc_nkb_dev(a.d);
                bn = reinterpret_cast<const float *>(
                         a.tc_rows + a.tc_row_blocks[a.nlist] * (int64_t)nkb * kTcBlockBytes) + T.blk0;
                // one product of the hi halves h(256 q), h(256 x) (fp16, round to
                // nearest: |256 q - h| <= 2^-11 |256 q| + 2^-25) differs from
                // <q, x> by at most 2^-10 (1 + 2^-11) sum |q_i x_i| + 2^-33 sqrt(d)
                // (|q| + |x|) (1 + 2^-11), and its fp32 accumulation of d exact
                // products by at most d 2^-24 sum |q_i x_i| (to nearest); the
                // margin takes 2^-10 + 2^-12 + d 2^-22 times |q| |x| (Cauchy-
                // Schwarz, with room for the norms' own rounding and an
                // accumulator that truncates) plus 2^-26 sqrt(d) (|q| + |x|)
                m_rel = 0.0009765625f + 0.000244140625f + (float)a.d * 2.384185791015625e-7f;
                m_abs = 1.4901161193847656e-8f * sqrtf((float)a.d);
                qn = valid ? a.qnorm[q] : 0.f;
                xn = xn_next = 0.f;
            }
        }
        __device__ void find_worst(int k) {
            wst_pos = 0;
            wst_s = KS(0);
            wst_id = KI(0);
            for (int j = 1; j < k; ++j) {
                const float s = KS(j);
                const long long id = KI(j);
                if (ranks_before(wst_s, wst_id, s, id)) {
                    wst_pos = j;
                    wst_s = s;
                    wst_id = id;
                }
            }
        }
        // one candidate row (s >= tau): self exclusion, then into the kept
        // list (appended while it has room, else in place of its last entry)
        __device__ __forceinline__ void take(const Args &a, const Tile &T, int64_t col, float sc) {
            if (a.k == kn && sc < wst_s) return;   // cannot rank before the last kept entry
            const long long id = ids_ch >= 0 ? ids_b[(ids_ch & 1) * tcb::kN + (col & (tcb::kN - 1))]
                                             : a.ids[T.r_begin + col];
            if (id == qid) return;
            insert(a, sc, id);
        }
        __device__ __forceinline__ void insert(const Args &a, float sc, long long id) {
            const int k = a.k;
            if (kn < k) {
                KS(kn) = sc;
                KI(kn) = id;
                if (++kn == k) find_worst(k);
                return;
            }
            if (!ranks_before(sc, id, wst_s, wst_id)) return;
            KS(wst_pos) = sc;
            KI(wst_pos) = id;
            find_worst(k);
        }
        // e holds 32 scores x `scale` (an exact power of two): the candidates
        __device__ __forceinline__ void select(const Args &a, const Tile &T, int64_t col0,
                                               const float (&e)[32], int ncol, float scale) {
            // a candidate needs s >= tau and, once k are kept, s >= the k-th
            // kept score (equal scores go on to the id tie-break)
            float thr = a.tau * scale;
            if (kn == a.k) thr = fmaxf(thr, wst_s * scale);
            // nearly every group has no candidate: one tree of maxima decides
            if (!(max_of_32(e) >= thr)) return;
            unsigned m = 0;
#pragma unroll
            for (int j = 0; j < 32; ++j) m |= (e[j] >= thr && j < ncol) ? (1u << j) : 0u;
            // one candidate at a time in a loop that is not unrolled: a single
            // copy of the insert, the score picked out of the registers
            const float inv = 1.f / scale;
            while (m) {
                const int j = __ffs(m) - 1;
                m &= m - 1u;
                take(a, T, col0 + j, pick32(e, j) * inv);
            }
        }
        // kScreen: v holds one-product scores x 2^16.  A row whose exact score
        // reaches the threshold (tau, or the last kept entry once k are kept)
        // has a screened score of at least the threshold minus the margin;
        // such rows, other than the query's own, are scored again by the
        // whole warp in fp32, one at a time, and only that score decides.
        // Every lane of the warp takes part (ncol is the same for all).
        __device__ __forceinline__ void screen(const Args &a, const Tile &T, int64_t col0,
                                               const float (&v)[32], int ncol) {
            if (ncol <= 0) return;
            float thr = a.tau;
            if (kn == a.k) thr = fmaxf(thr, wst_s);
            const float cut = (thr - (m_rel * qn * xn + m_abs * (qn + xn))) * 65536.f;
            const bool any = valid && max_of_32(v) >= cut;
            if (!__any_sync(0xffffffffu, any)) return;
            unsigned m = 0;
            if (any) {
#pragma unroll
                for (int j = 0; j < 32; ++j) m |= (v[j] >= cut && j < ncol) ? (1u << j) : 0u;
                // the query's own row leaves here (ids from the warp's copy)
                const long long *cid = ids_b + (ids_ch & 1) * tcb::kN + (col0 & (tcb::kN - 1));
                for (unsigned mm = m; mm; mm &= mm - 1u) {
                    const int j = __ffs(mm) - 1;
                    if (cid[j] == qid) m &= ~(1u << j);
                }
            }
            // up to four candidates at a time, one from each of the first four
            // lanes that have one, each scored by eight lanes (lane-strided
            // fused multiply-adds, all loads in flight, then a butterfly sum
            // over the eight)
            const int lane = (int)(threadIdx.x & 31u), sub = lane >> 3;
            for (;;) {
                unsigned lanes = __ballot_sync(0xffffffffu, m != 0u);
                if (!lanes) break;
                int own = -1;   // which of the batch's pairs this lane owns
                int Lg = 0, jg = 0, npick = 0;
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    if (!lanes) break;
                    const int L = __ffs(lanes) - 1;
                    lanes &= lanes - 1u;
                    const int j = __ffs(__shfl_sync(0xffffffffu, m, L)) - 1;
                    if (lane == L) own = g;
                    if (sub == g) {
                        Lg = L;
                        jg = j;
                    }
                    ++npick;
                }
                const int qL = __shfl_sync(0xffffffffu, q, Lg);
                float acc = 0.f;
                if (sub < npick) {   // d <= 256: at most 8 float4 of each row per lane, all in flight
                    const float *u = a.Q + (int64_t)qL * a.d;
                    const float *w = a.X + (T.r_begin + col0 + jg) * a.d;
                    float4 x[8], y[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int c = 4 * (lane & 7) + 32 * i;
                        x[i] = c < a.d ? __ldg(reinterpret_cast<const float4 *>(u + c)) : make_float4(0.f, 0.f, 0.f, 0.f);
                        y[i] = c < a.d ? __ldg(reinterpret_cast<const float4 *>(w + c)) : make_float4(0.f, 0.f, 0.f, 0.f);
                    }
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        acc = fmaf(x[i].x, y[i].x, acc);
                        acc = fmaf(x[i].y, y[i].y, acc);
                        acc = fmaf(x[i].z, y[i].z, acc);
                        acc = fmaf(x[i].w, y[i].w, acc);
                    }
                }
#pragma unroll
                for (int o = 4; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                // lane L of pair g reads the sum of sub-group g
                const float sc = __shfl_sync(0xffffffffu, acc, own >= 0 ? 8 * own : 0);
                if (own >= 0) {
                    const int j = __ffs(m) - 1;
                    m &= m - 1u;
                    if (sc >= a.tau && !(kn == a.k && sc < wst_s))
                        insert(a, sc, ids_b[(ids_ch & 1) * tcb::kN + (col0 & (tcb::kN - 1)) + j]);
                }
            }
        }
        // the row ids of chunk c into buffer c % 2 of this warp (8-byte
        // asynchronous copies, one group)
        __device__ __forceinline__ void copy_ids(const Args &a, const Tile &T, int c) {
            const int64_t r0 = T.r_begin + (int64_t)c * tcb::kN;
            const int64_t left = T.nb - (int64_t)c * tcb::kN;
            const int nrow = left < tcb::kN ? (int)left : tcb::kN;
            long long *dst = ids_b + (c & 1) * tcb::kN;
            for (int j = slot & 31; j < nrow; j += 32)
                asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(tc::smem_u32(dst + j)),
                             "l"(a.ids + r0 + j)
                             : "memory");
            asm volatile("cp.async.commit_group;\n" ::: "memory");
        }
        // Before chunk ch's accumulator wait (bulk pipeline): copies in flight
        // for it -- kRQ, the chunk's factors into this warp's shared copy (one
        // coalesced 512-byte copy per warp); the row ids one chunk ahead (both
        // of the first two chunks at ch = 0), so their latency hides behind a
        // chunk; kScreen, the block norm of the next chunk into a register.
        // Every lane of the warp is done with the buffers being refilled (the
        // chunk before last).
        __device__ __forceinline__ void prefetch(const Args &a, const Tile &T, int ch) {
            const int nch = (int)ceil_div(T.nb, tcb::kN);
            __syncwarp();
            if (ch == 0) copy_ids(a, T, 0);
            if constexpr (kRQ) {
                const float *src = T.fac + (int64_t)ch * tcb::kN + 4 * (slot & 31);
                const uint32_t dst = tc::smem_u32(fs + 4 * (slot & 31));
                asm volatile("cp.async.ca.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
                asm volatile("cp.async.commit_group;\n" ::: "memory");
            }
            if (ch + 1 < nch) copy_ids(a, T, ch + 1);
            if constexpr (kScreen) {
                xn = ch == 0 ? bn[0] : xn_next;
                xn_next = ch + 1 < nch ? bn[ch + 1] : 0.f;
            }
        }
        // after the accumulator wait: every group but the next chunk's ids
        // has landed
        __device__ __forceinline__ void start(const Args &, const Tile &T, int ch) {
            if (ch + 1 < (int)ceil_div(T.nb, tcb::kN))
                asm volatile("cp.async.wait_group 1;\n" ::: "memory");
            else
                asm volatile("cp.async.wait_group 0;\n" ::: "memory");
            __syncwarp();
            ids_ch = ch;
        }
        // v holds the chunk's raw accumulator values: exact, similarities x
        // 2^16; kRQ, <u - mid, q'> x 2^8 (the codes are not scaled)
        __device__ void chunk(const Args &a, const Tile &T, int64_t col0, const float (&v)[32],
                              int ncol) {
            if constexpr (kScreen) {
                screen(a, T, col0, v, ncol);
                return;
            }
            if (!valid || ncol <= 0) return;
            if constexpr (kRQ) {
                // the estimates qc + f <u - mid, q'> (the factor copy holds
                // f x 2^-8, the scale of the accumulator: one fma each) against
                // the threshold, straight into a mask; the rare candidates
                // compute theirs again, with the same arithmetic
                const float4 *f4 = reinterpret_cast<const float4 *>(fs + (col0 & (tcb::kN - 1)));
                float thr = a.tau;
                if (kn == a.k) thr = fmaxf(thr, wst_s);
                unsigned m = 0;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float4 f = f4[j];
                    m |= (fmaf(f.x, v[4 * j], qc) >= thr) ? 1u << (4 * j) : 0u;
                    m |= (fmaf(f.y, v[4 * j + 1], qc) >= thr) ? 2u << (4 * j) : 0u;
                    m |= (fmaf(f.z, v[4 * j + 2], qc) >= thr) ? 4u << (4 * j) : 0u;
                    m |= (fmaf(f.w, v[4 * j + 3], qc) >= thr) ? 8u << (4 * j) : 0u;
                }
                if (ncol < 32) m &= (1u << ncol) - 1u;
                while (m) {
                    const int j = __ffs(m) - 1;
                    m &= m - 1u;
                    take(a, T, col0 + j, fmaf(fs[(col0 & (tcb::kN - 1)) + j], pick32(v, j), qc));
                }
            } else {
                select(a, T, col0, v, ncol, 65536.f);
            }
        }
        __device__ void end(const Args &a, const Tile &T) {
            if (valid) {
                const int k = a.k;
                for (int j = 1; j < kn; ++j) {   // the list in result order (insertion sort)
                    const float s = KS(j);
                    const long long id = KI(j);
                    int i = j;
                    while (i > 0 && ranks_before(s, id, KS(i - 1), KI(i - 1))) {
                        KS(i) = KS(i - 1);
                        KI(i) = KI(i - 1);
                        --i;
                    }
                    KS(i) = s;
                    KI(i) = id;
                }
                for (int j = 0; j < kn; ++j) {
                    a.res_s[(int64_t)item * k + j] = KS(j);
                    a.res_id[(int64_t)item * k + j] = KI(j);
                }
                a.res_cnt[item] = kn;
                if (kn > 0) {   // a hit at rank j commits ranks up to min(j + W, nprobe)
                    const long long reach = (long long)rank + a.W;
                    atomicMax(&a.S[q], reach < a.nprobe ? (int)reach : a.nprobe);
                }
            }
            if (slot == 0) {   // one epilogue thread per tile counts the work
                atomicAdd(&a.ctl->tot_rows, (unsigned long long)T.nb);
                atomicAdd(&a.ctl->tot_pairs, (unsigned long long)T.nb * (unsigned long long)T.ni);
                atomicAdd(&a.ctl->tot_rows_tc, (unsigned long long)T.nb);
                atomicAdd(&a.ctl->tot_pairs_tc, (unsigned long long)T.nb * (unsigned long long)T.ni);
            }
        }
    };
};
static_assert(tcb::has_epi_wait<ScanModeT<false>>::value && tcb::has_epi_wait<ScanModeT<false, true>>::value,
              "the scan's epilogue wait takes the search's wait_limit");

using ScanMode = ScanModeT<false>;
using ScanModeRQ = ScanModeT<true>;
using ScanModeScreen = ScanModeT<false, true>;

bool scan_tc_fits(int k) { return scan_tc_smem_bytes(k) <= (size_t)(232448 - 128); }

size_t scan_tc_smem_bytes(int k) {
    return tcp::Geometry<ScanMode::kN>::smem_bytes((size_t)tcp::kM * k * (sizeof(float) + sizeof(long long)));
}

__global__ void __launch_bounds__(tcp::kThreads, 1) k_scan_tc(SearchArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcp::run_pipeline<ScanMode>(a, smem_raw);
}

// the kept lists, the factor copies (the scan over codes) and the row-id
// buffers (two per epilogue warp)
static size_t scan_epi_bytes(int k) {
    return (size_t)tcp::kM * k * (sizeof(float) + sizeof(long long)) + kEpiFacBytes + kEpiIdsBytes;
}

int scan_bulk_stages(int d, int k) {
    return tcb::stages_for((int)ceil_div(d, 64), scan_epi_bytes(k), 232448 - 128);
}

__global__ void __launch_bounds__(tcb::kThreads, 1) k_scan_bulk(SearchArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<ScanMode>(a, smem_raw, a.tc_stages);
}

cudaError_t prepare_scan_bulk(int d, int k, int stages) {
    return cudaFuncSetAttribute(k_scan_bulk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)tcb::smem_bytes(stages, scan_epi_bytes(k)));
}

// the screening scan: stages of two 16 KB K-blocks (the hi halves)
constexpr int kScreenStagesMax = 6;
static size_t scan_screen_epi_bytes(int k) { return scan_epi_bytes(k); }

int scan_screen_stages(int d, int k) {
    return tcb::stages_for((int)ceil_div(d, 64), scan_screen_epi_bytes(k), 232448 - 128,
                           tcb::kStageBytesHi, kScreenStagesMax);
}

__global__ void __launch_bounds__(tcb::kThreads, 1) k_scan_screen(SearchArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<ScanModeScreen>(a, smem_raw, a.tc_stages);
}

cudaError_t prepare_scan_screen(int d, int k, int stages) {
    return cudaFuncSetAttribute(k_scan_screen, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)tcb::smem_bytes(stages, scan_screen_epi_bytes(k), tcb::kStageBytesHi));
}

void enqueue_scan_bulk(const SearchArgs &a, cudaStream_t st) {
    if (a.tc_screen)
        k_scan_screen<<<num_sms(), tcb::kThreads,
                        tcb::smem_bytes(a.tc_stages, scan_screen_epi_bytes(a.k), tcb::kStageBytesHi), st>>>(a);
    else
        k_scan_bulk<<<num_sms(), tcb::kThreads,
                      tcb::smem_bytes(a.tc_stages, scan_epi_bytes(a.k)), st>>>(a);
}

// the scan over codes: stages of two 16 KB K-blocks
static size_t scan_rq_epi_bytes(int k) { return scan_epi_bytes(k); }

int scan_rq_stages(int d, int k) {
    return tcb::stages_for((int)ceil_div(d, 64), scan_rq_epi_bytes(k), 232448 - 128, tcb::kStageBytesHi);
}

__global__ void __launch_bounds__(tcb::kThreads, 1) k_scan_rq(SearchArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<ScanModeRQ>(a, smem_raw, a.tc_stages);
}

cudaError_t prepare_scan_rq(int d, int k, int stages) {
    return cudaFuncSetAttribute(k_scan_rq, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)tcb::smem_bytes(stages, scan_rq_epi_bytes(k), tcb::kStageBytesHi));
}

void enqueue_scan_rq(const SearchArgs &a, cudaStream_t st) {
    k_scan_rq<<<num_sms(), tcb::kThreads, tcb::smem_bytes(a.tc_stages, scan_rq_epi_bytes(a.k), tcb::kStageBytesHi),
                st>>>(a);
}

cudaError_t prepare_scan_tc(int k) {
    return cudaFuncSetAttribute(k_scan_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)scan_tc_smem_bytes(k));
}

void enqueue_scan_tc(const SearchArgs &a, cudaStream_t st) {
    k_scan_tc<<<num_sms(), tcp::kThreads, scan_tc_smem_bytes(a.k), st>>>(a);
}

}  // namespace sieve
