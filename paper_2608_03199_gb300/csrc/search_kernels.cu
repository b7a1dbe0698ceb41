// search_kernels.cu -- the rounds of the threshold-aware IVF search (sm_103a).
//
// One round (continuous batching, Sec. 4.2 / Algorithm 1; lookahead,
// Sec. 4.3 / Algorithm 2):
//   k_issue    every query with committed, not yet issued ranks e..s emits
//              (query, rank) items: one per round without lookahead, all of
//              them with lookahead; the partition of each item is counted
//   k_bucket   one block: prefix sums of the per-partition counts give the
//              ready queue as a CSR of partition groups, cut into tiles of at
//              most QT items (the microbatches of Sec. 4.2)
//   k_scatter  items are placed in their partition group
//   k_scan     persistent blocks take tiles: the group's queries x all rows
//              of the partition, the tau test, the local top-k per item and,
//              on a hit at rank j, stop line s = max(s, min(j + W, nprobe))
//   k_merge    each query folds its items' local results into its top-k
//              (MergeTopK) and reports whether committed ranks remain
//   k_round_end decides whether another round runs (the WHILE condition of
//              the device-resident round loop) and resets the counters
#include "search.cuh"

namespace sieve {

// ---------------------------------------------------------------------------
__global__ void k_init(SearchArgs a) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int s0 = a.W < a.nprobe ? a.W : a.nprobe;   // initial stop line min(W, nprobe)
    for (int64_t q = t0; q < a.nq; q += stride) {
        a.S[q] = s0;
        a.E[q] = 1;
        a.out_count[q] = 0;
    }
    for (int64_t i = t0; i < a.nq * a.k; i += stride) {
        a.out_ids[i] = -1;
        a.out_scores[i] = -__int_as_float(0x7f800000);
        if (a.out_rank) a.out_rank[i] = 0;
    }
    if (a.hit_bits)
        for (int64_t i = t0; i < a.nq * a.hit_words; i += stride) a.hit_bits[i] = 0u;
    // the control block was zeroed by a memset before this kernel; a list
    // offset table that is not a partition of [0, n) is reported and the
    // search then issues nothing
    for (int64_t p = t0; p < a.nlist; p += stride) {
        a.counts[p] = 0;
        const int64_t lo = a.off[p], hi = a.off[p + 1];
        if (lo < 0 || hi < lo || hi > a.n || (p == 0 && lo != 0) || (p == a.nlist - 1 && hi != a.n))
            atomicExch(&a.ctl->status, SIEVE_EINVAL);
    }
}

// the queries' Euclidean norms for the screening scan's error bound: a warp
// per query, lane-strided fp32 sums of squares and a butterfly sum
__global__ void k_qnorm(SearchArgs a) {
    const int lane = (int)lane_id();
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t q = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; q < a.nq; q += warps) {
        const float *row = a.Q + q * a.d;
        float ss = 0.f;
        for (int c = 4 * lane; c < a.d; c += 128) {
            const float4 x = __ldg(reinterpret_cast<const float4 *>(row + c));
            ss = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, fmaf(x.w, x.w, ss))));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) a.qnorm[q] = sqrtf(ss);
    }
}

__global__ void k_finalize(SearchArgs a) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < a.nq; q += stride)
        a.out_probes[q] = a.S[q];
}

// ---------------------------------------------------------------------------
// exclusive block scan of one int per thread (blockDim.x == kIssueThreads)
constexpr int kIssueThreads = 256;

__device__ __forceinline__ int block_exclusive_scan(int v, int *warp_tot, int *total) {
    const unsigned lane = lane_id(), warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= (unsigned)o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < kIssueThreads / 32 ? warp_tot[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= (unsigned)o) w += y;
        }
        if (lane < kIssueThreads / 32) warp_tot[lane] = w;   // inclusive warp prefix
        if (lane == kIssueThreads / 32 - 1) *total = w;
    }
    __syncthreads();
    int before = warp > 0 ? warp_tot[warp - 1] : 0;
    int r = before + x - v;
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(kIssueThreads) k_issue(SearchArgs a) {
    __shared__ int warp_tot[kIssueThreads / 32];
    __shared__ int tot_items, tot_act, base_items, base_act;
    Ctl *ctl = a.ctl;
    const int64_t cap = a.cap;
    if (*(volatile int *)&ctl->status != 0) return;   // bad input: issue nothing
    for (int64_t q0 = (int64_t)blockIdx.x * kIssueThreads; q0 < a.nq;
         q0 += (int64_t)gridDim.x * kIssueThreads) {
        const int64_t q = q0 + threadIdx.x;
        int want = 0, e = 0;
        if (q < a.nq) {
            int s = a.S[q];
            e = a.E[q];
            if (e <= s) want = a.lookahead ? s - e + 1 : 1;
        }
        int off = block_exclusive_scan(want, warp_tot, &tot_items);
        int aoff = block_exclusive_scan(want > 0 ? 1 : 0, warp_tot, &tot_act);
        if (threadIdx.x == 0) {
            base_items = tot_items ? atomicAdd(&ctl->n_items, tot_items) : 0;
            base_act = tot_act ? atomicAdd(&ctl->n_active, tot_act) : 0;
        }
        __syncthreads();
        if (want > 0) {
            int64_t start = (int64_t)base_items + off;
            int64_t room = cap - start;
            int got = room <= 0 ? 0 : (room < want ? (int)room : want);
            if (got < want) atomicAdd(&ctl->n_deferred, 1);
            const int32_t *ord = a.order + q * a.nprobe;
            for (int r = 0; r < got; ++r) {
                int64_t idx = start + r;
                int rank = e + r;
                int p = ord[rank - 1];
                if (p < 0 || p >= a.nlist) {   // a caller-supplied order out of range
                    atomicExch(&ctl->status, SIEVE_EINVAL);
                    p = 0;
                }
                a.item_q[idx] = (int)q;
                a.item_rank[idx] = rank;
                a.item_p[idx] = p;
                atomicAdd(&a.counts[p], 1);
            }
            a.E[q] = e + got;
            a.active[base_act + aoff] = make_int4((int)q, (int)(got > 0 ? start : 0), got, 0);
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
constexpr int kBucketThreads = 1024;

// A group of c items is cut into chunks of up to kTcTile; a chunk with at
// least tc_min items is one tensor-core tile, a smaller one is cut into SIMT
// tiles of up to QT items.
__device__ __forceinline__ void count_tiles(int c, int tc_min, int serial, int &n_tc, int &n_simt) {
    n_tc = 0;
    n_simt = 0;
    if (serial) {   // serial traversal: one tile per item, no regrouping across queries
        if (tc_min > 0) n_tc = c;
        else n_simt = c;
        return;
    }
    for (int o = 0; o < c; o += kTcTile) {
        const int sz = c - o < kTcTile ? c - o : kTcTile;
        if (tc_min > 0 && sz >= tc_min)
            ++n_tc;
        else
            n_simt += (sz + QT - 1) / QT;
    }
}

// Tensor-core tiles are listed longest first (by the partition's 128-row
// chunks, capped), so the blocks that draw them from the work counter finish
// together; the tiles of one partition stay adjacent.
constexpr int kTileClasses = 128;
__device__ __forceinline__ int tile_class(const SearchArgs &a, int64_t p) {
    const int64_t ch = ceil_div(a.off[p + 1] - a.off[p], kTcTile);
    return ch < kTileClasses - 1 ? (int)ch : kTileClasses - 1;
}

__global__ void __launch_bounds__(kBucketThreads) k_bucket(SearchArgs a) {
    __shared__ int warp_tot[32];
    __shared__ int sums[3];
    __shared__ int cls[kTileClasses];   // tensor-core tiles per class, then class cursors
    Ctl *ctl = a.ctl;
    const int64_t nl = a.nlist;
    const int per = (int)ceil_div(nl, kBucketThreads);
    const int64_t p0 = (int64_t)threadIdx.x * per;
    for (int i = threadIdx.x; i < kTileClasses; i += blockDim.x) cls[i] = 0;
    __syncthreads();
    int my[3] = {0, 0, 0};   // items, SIMT tiles, tensor-core tiles
    int my_groups = 0;
    for (int64_t p = p0; p < p0 + per && p < nl; ++p) {
        const int c = a.counts[p];
        int ntc, ns;
        count_tiles(c, a.tc_min, a.serial, ntc, ns);
        my[0] += c;
        my[1] += ns;
        my[2] += ntc;
        my_groups += c > 0;
        if (ntc) atomicAdd(&cls[tile_class(a, p)], ntc);
    }
    // three exclusive scans over threads
    const unsigned lane = lane_id(), warp = threadIdx.x >> 5;
    int ex[3];
    for (int v = 0; v < 3; ++v) {
        int x = my[v];
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= (unsigned)o) x += y;
        }
        if (lane == 31) warp_tot[warp] = x;
        __syncthreads();
        if (warp == 0) {
            int w = warp_tot[lane];
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= (unsigned)o) w += y;
            }
            warp_tot[lane] = w;
            if (lane == 31) sums[v] = w;
        }
        __syncthreads();
        ex[v] = (warp > 0 ? warp_tot[warp - 1] : 0) + x - my[v];
        __syncthreads();
    }
    if (threadIdx.x == 0) {   // class cursors: exclusive scan, longest class first
        int run = 0;
        for (int i = kTileClasses - 1; i >= 0; --i) {
            const int v = cls[i];
            cls[i] = run;
            run += v;
        }
    }
    __syncthreads();
    int ioff = ex[0], soff = ex[1];
    for (int64_t p = p0; p < p0 + per && p < nl; ++p) {
        const int c = a.counts[p];
        a.cursor[p] = ioff;
        int ntc, ns;
        count_tiles(c, a.tc_min, a.serial, ntc, ns);
        int toff = ntc ? atomicAdd(&cls[tile_class(a, p)], ntc) : 0;
        if (a.serial) {   // one tile per item
            for (int o = 0; o < c; ++o) {
                if (a.tc_min > 0)
                    a.tc_tiles[toff++] = make_int4((int)p, ioff + o, 1, 0);
                else
                    a.tiles[soff++] = make_int4((int)p, ioff + o, 1, 0);
            }
            ioff += c;
            a.counts[p] = 0;
            continue;
        }
        for (int o = 0; o < c; o += kTcTile) {
            const int sz = c - o < kTcTile ? c - o : kTcTile;
            if (a.tc_min > 0 && sz >= a.tc_min) {
                a.tc_tiles[toff++] = make_int4((int)p, ioff + o, sz, 0);
            } else {
                for (int u = 0; u < sz; u += QT)
                    a.tiles[soff++] = make_int4((int)p, ioff + o + u, sz - u < QT ? sz - u : QT, 0);
            }
        }
        ioff += c;
        a.counts[p] = 0;   // ready for the next round's issue
    }
    // groups: reduce
    int g = my_groups;
    for (int o = 16; o > 0; o >>= 1) g += __shfl_down_sync(0xffffffffu, g, o);
    if (lane == 0 && g) atomicAdd(&ctl->tot_groups, (unsigned long long)g);
    if (threadIdx.x == 0) {
        ctl->n_tiles = sums[1];
        ctl->n_tc_tiles = sums[2];
        ctl->tile_next = 0;
        ctl->tc_tile_next = 0;
    }
}

__global__ void k_scatter(SearchArgs a) {
    const int64_t n = a.ctl->n_items < a.cap ? a.ctl->n_items : a.cap;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        int pos = atomicAdd(&a.cursor[a.item_p[i]], 1);
        a.bucketed[pos] = (int)i;
    }
}

// ---------------------------------------------------------------------------
// the grouped contraction with the fused tau / top-k / stop-line epilogue
constexpr int kPool = 256;   // candidate staging entries per block

struct PoolEntry {
    float s;
    int slot;
    long long id;
};

size_t scan_smem_bytes(int d, int k) {
    size_t dpad = (size_t)round_up(d, DK);
    size_t b = 0;
    b += (size_t)QT * (dpad + 4) * sizeof(float);   // Qs
    b += 2ull * RT * LDX * sizeof(float);            // Xs (2 stages)
    b += (size_t)kPool * sizeof(PoolEntry);          // pool
    b += (size_t)QT * k * sizeof(long long);         // kept ids
    b += (size_t)QT * k * sizeof(float);             // kept scores
    b = round_up(b, 16);
    return b;
}

__global__ void __launch_bounds__(kThreads) k_scan(SearchArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int s_tile, s_pool_n;
    __shared__ int slot_item[QT], slot_q[QT], slot_rank[QT], kept_n[QT];
    __shared__ long long slot_qid[QT];

    const int d = a.d, k = a.k;
    const int dpad = (int)round_up(d, DK);
    const int ldq = dpad + 4;
    float *Qs = reinterpret_cast<float *>(smem_raw);
    float *Xs = Qs + QT * ldq;
    PoolEntry *pool = reinterpret_cast<PoolEntry *>(Xs + 2 * RT * LDX);
    long long *kept_id = reinterpret_cast<long long *>(pool + kPool);
    float *kept_s = reinterpret_cast<float *>(kept_id + QT * k);

    const int tid = threadIdx.x;
    const int tq = tid & 7, tr = tid >> 3;
    const unsigned lane = lane_id(), warp = tid >> 5;
    const float tau = a.tau;
    Ctl *ctl = a.ctl;
    const int n_tiles = ctl->n_tiles;

    if (tid == 0) s_pool_n = 0;
    for (;;) {
        if (tid == 0) s_tile = atomicAdd(&ctl->tile_next, 1);
        __syncthreads();
        const int t = s_tile;
        if (t >= n_tiles) break;
        const int4 tile = a.tiles[t];
        const int p = tile.x, ib = tile.y, ni = tile.z;
        if (tid < QT) {
            kept_n[tid] = 0;
            if (tid < ni) {
                int item = a.bucketed[ib + tid];
                int q = a.item_q[item];
                slot_item[tid] = item;
                slot_q[tid] = q;
                slot_rank[tid] = a.item_rank[item];
                slot_qid[tid] = a.qids ? a.qids[q] : (long long)-0x7fffffffffffffffll - 1;
            }
        }
        __syncthreads();
        // gathered queries of the group -> Qs[QT][ldq] (zero past ni and past d)
        const int nv = dpad / 4;
        for (int idx = tid; idx < QT * nv; idx += kThreads) {
            int i = idx / nv, v = idx % nv;
            float4 val = make_float4(0.f, 0.f, 0.f, 0.f);
            if (i < ni && 4 * v < d)
                val = *reinterpret_cast<const float4 *>(a.Q + (int64_t)slot_q[i] * d + 4 * v);
            *reinterpret_cast<float4 *>(Qs + i * ldq + 4 * v) = val;
        }
        const int64_t r_begin = a.off[p];
        const int64_t np = a.off[p + 1] - r_begin;
        const float *part = a.X + r_begin * d;
        const int nch = dpad / DK;
        const int64_t nsteps = ceil_div(np, RT) * nch;
        float acc[4][4];
        if (nsteps > 0) {
            stage_rows(Xs, part, np, d, 0, 0);
            cp_async_commit();
        }
        for (int64_t s = 0; s < nsteps; ++s) {
            const int64_t rt = s / nch;
            const int c = (int)(s % nch);
            if (s + 1 < nsteps) {
                const int64_t s1 = s + 1;
                stage_rows(Xs + ((s1 & 1) ? RT * LDX : 0), part, np, d, (s1 / nch) * RT,
                           (int)(s1 % nch) * DK);
                cp_async_commit();
                cp_async_wait<1>();
            } else {
                cp_async_wait<0>();
            }
            __syncthreads();
            if (c == 0) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
            }
            contract_chunk(acc, Qs, ldq, c * DK, Xs + ((s & 1) ? RT * LDX : 0), tq, tr);
            if (c == nch - 1) {
                // ---- epilogue of row tile rt: tau test, self exclusion, staging ----
                unsigned mask = 0;
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        int slot = tq + 8 * i;
                        int64_t r = rt * RT + tr + 16 * j;
                        if (slot < ni && r < np && acc[i][j] >= tau) mask |= 1u << (4 * i + j);
                    }
                if (__syncthreads_or(mask != 0)) {
                    long long idv[16];
#pragma unroll
                    for (int b = 0; b < 16; ++b) {
                        idv[b] = 0;
                        if (mask & (1u << b)) {
                            int slot = tq + 8 * (b >> 2);
                            int64_t r = rt * RT + tr + 16 * (b & 3);
                            idv[b] = a.ids[r_begin + r];
                            if (idv[b] == slot_qid[slot]) mask &= ~(1u << b);
                        }
                    }
                    for (;;) {
#pragma unroll
                        for (int b = 0; b < 16; ++b) {
                            if (mask & (1u << b)) {
                                int pos = atomicAdd(&s_pool_n, 1);
                                if (pos < kPool) {
                                    pool[pos].s = acc[b >> 2][b & 3];
                                    pool[pos].slot = tq + 8 * (b >> 2);
                                    pool[pos].id = idv[b];
                                    mask &= ~(1u << b);
                                }
                            }
                        }
                        __syncthreads();
                        // flush: warp w owns slots w, w+4, ...
                        const int pn = s_pool_n < kPool ? s_pool_n : kPool;
                        for (int base = 0; base < pn; base += 32) {
                            int e = base + (int)lane;
                            bool mine = e < pn && (pool[e].slot & 3) == (int)warp;
                            unsigned bal = __ballot_sync(0xffffffffu, mine);
                            while (bal) {
                                int src = __ffs(bal) - 1;
                                bal &= bal - 1;
                                const PoolEntry pe = pool[base + src];
                                warp_list_insert(kept_s + pe.slot * k, kept_id + pe.slot * k,
                                                 &kept_n[pe.slot], k, pe.s, pe.id);
                            }
                        }
                        __syncthreads();
                        if (tid == 0) s_pool_n = 0;
                        if (!__syncthreads_or(mask != 0)) break;
                    }
                }
            }
            __syncthreads();
        }
        // ---- per-item local results and the stop-line update ----
        for (int slot = warp; slot < ni; slot += kThreads / 32) {
            const int item = slot_item[slot];
            const int n = kept_n[slot];
            for (int j = lane; j < n; j += 32) {
                a.res_s[(int64_t)item * k + j] = kept_s[slot * k + j];
                a.res_id[(int64_t)item * k + j] = kept_id[slot * k + j];
            }
            if (lane == 0) {
                a.res_cnt[item] = n;
                if (n > 0) {   // a hit at rank j commits ranks up to min(j + W, nprobe)
                    long long reach = (long long)slot_rank[slot] + a.W;
                    int line = reach < a.nprobe ? (int)reach : a.nprobe;
                    atomicMax(&a.S[slot_q[slot]], line);
                }
            }
        }
        if (tid == 0) {
            atomicAdd(&ctl->tot_rows, (unsigned long long)np);
            atomicAdd(&ctl->tot_pairs, (unsigned long long)np * (unsigned long long)ni);
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// MergeTopK: one warp per query of this round; the running top-k lives in the
// output arrays (sorted), two entries per lane.
constexpr int kMergeThreads = 256;

__global__ void __launch_bounds__(kMergeThreads) k_merge(SearchArgs a) {
    Ctl *ctl = a.ctl;
    const int n_act = ctl->n_active;
    const int k = a.k;
    const unsigned lane = lane_id();
    const int64_t gw = ((int64_t)blockIdx.x * kMergeThreads + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * kMergeThreads) >> 5;
    const float ninf = -__int_as_float(0x7f800000);
    for (int64_t w = gw; w < n_act; w += nw) {
        const int4 act = a.active[w];
        const int q = act.x, start = act.y, got = act.z;
        int n = a.out_count[q];
        float r0s = ninf, r1s = ninf;
        long long r0i = -1, r1i = -1;
        int r0r = 0, r1r = 0;   // provenance ranks (kept only when out_rank is set)
        const int64_t ob = (int64_t)q * k;
        if ((int)lane < n) { r0s = a.out_scores[ob + lane]; r0i = a.out_ids[ob + lane]; }
        if ((int)lane + 32 < n) { r1s = a.out_scores[ob + lane + 32]; r1i = a.out_ids[ob + lane + 32]; }
        if (a.out_rank) {
            if ((int)lane < n) r0r = a.out_rank[ob + lane];
            if ((int)lane + 32 < n) r1r = a.out_rank[ob + lane + 32];
        }
        bool changed = false;
        for (int it = start; it < start + got; ++it) {
            const int c = a.res_cnt[it];
            const int rk = a.item_rank[it];
            if (a.hit_bits && c > 0 && lane == 0)   // this query's items: one warp, no race
                a.hit_bits[(int64_t)q * a.hit_words + (rk - 1) / 32] |= 1u << ((rk - 1) % 32);
            for (int j = 0; j < c; ++j) {
                const float s = a.res_s[(int64_t)it * k + j];
                const long long id = a.res_id[(int64_t)it * k + j];
                bool b0 = (int)lane < n && ranks_before(r0s, r0i, s, id);
                bool b1 = (int)lane + 32 < n && ranks_before(r1s, r1i, s, id);
                int pos = __popc(__ballot_sync(0xffffffffu, b0)) +
                          __popc(__ballot_sync(0xffffffffu, b1));
                if (pos >= k) break;   // the rest of this sorted list ranks lower
                float u0s = __shfl_up_sync(0xffffffffu, r0s, 1);
                long long u0i = __shfl_up_sync(0xffffffffu, r0i, 1);
                float u1s = __shfl_up_sync(0xffffffffu, r1s, 1);
                long long u1i = __shfl_up_sync(0xffffffffu, r1i, 1);
                float w31s = __shfl_sync(0xffffffffu, r0s, 31);
                long long w31i = __shfl_sync(0xffffffffu, r0i, 31);
                int u0r = __shfl_up_sync(0xffffffffu, r0r, 1);
                int u1r = __shfl_up_sync(0xffffffffu, r1r, 1);
                const int w31r = __shfl_sync(0xffffffffu, r0r, 31);
                if (lane == 0) { u1s = w31s; u1i = w31i; u1r = w31r; }
                const int j0 = lane, j1 = lane + 32;
                if (j0 == pos) { r0s = s; r0i = id; r0r = rk; }
                else if (j0 > pos) { r0s = u0s; r0i = u0i; r0r = u0r; }
                if (j1 == pos) { r1s = s; r1i = id; r1r = rk; }
                else if (j1 > pos) { r1s = u1s; r1i = u1i; r1r = u1r; }
                n = n < k ? n + 1 : k;
                changed = true;
            }
        }
        if (changed) {
            if ((int)lane < k) {
                a.out_scores[ob + lane] = (int)lane < n ? r0s : ninf;
                a.out_ids[ob + lane] = (int)lane < n ? r0i : -1;
            }
            if ((int)lane + 32 < k) {
                a.out_scores[ob + lane + 32] = (int)lane + 32 < n ? r1s : ninf;
                a.out_ids[ob + lane + 32] = (int)lane + 32 < n ? r1i : -1;
            }
            if (a.out_rank) {
                if ((int)lane < k) a.out_rank[ob + lane] = (int)lane < n ? r0r : 0;
                if ((int)lane + 32 < k) a.out_rank[ob + lane + 32] = (int)lane + 32 < n ? r1r : 0;
            }
            if (lane == 0) a.out_count[q] = n;
        }
        if (lane == 0 && a.E[q] <= a.S[q]) atomicAdd(&ctl->n_continue, 1);
    }
}

// ---------------------------------------------------------------------------
__global__ void k_round_end(SearchArgs a, cudaGraphConditionalHandle cond, int use_cond) {
    Ctl *c = a.ctl;
    const int items = c->n_items < a.cap ? c->n_items : (int)a.cap;
    c->tot_items += (unsigned long long)items;
    c->tot_tiles += (unsigned long long)(c->n_tiles + c->n_tc_tiles);
    c->round += 1;
    int more = (c->n_continue > 0 || c->n_deferred > 0) && c->status == 0 ? 1 : 0;
    if (more && c->round >= a.max_rounds) {
        c->status = SIEVE_ELIMIT;
        more = 0;
    }
    c->more = more;
    c->n_items = 0;
    c->n_active = 0;
    c->n_tiles = 0;
    c->n_tc_tiles = 0;
    c->tile_next = 0;
    c->tc_tile_next = 0;
    c->n_deferred = 0;
    c->n_continue = 0;
    if (use_cond) cudaGraphSetConditional(cond, more ? 1u : 0u);
}

// ---------------------------------------------------------------------------
// host-side launch helpers

int num_sms() {
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    return sms;
}

cudaError_t prepare_scan_kernel(size_t smem) {
    return cudaFuncSetAttribute(k_scan, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

cudaError_t launch_init(const SearchArgs &a, cudaStream_t st) {
    int64_t work = a.nq * a.k > a.nlist ? a.nq * a.k : a.nlist;
    int blocks = (int)std::min<int64_t>(ceil_div(work > 0 ? work : 1, 256), 4 * num_sms());
    cudaError_t e = cudaMemsetAsync(a.ctl, 0, sizeof(Ctl), st);
    if (e != cudaSuccess) return e;
    k_init<<<blocks, 256, 0, st>>>(a);
    if (a.tc_screen && a.nq > 0)
        k_qnorm<<<(int)std::min<int64_t>(ceil_div(a.nq, 8), 16 * num_sms()), 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_finalize(const SearchArgs &a, cudaStream_t st) {
    int blocks = (int)std::min<int64_t>(ceil_div(a.nq, 256), 4 * num_sms());
    k_finalize<<<blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_round(const SearchArgs &a, size_t scan_smem, int scan_blocks,
                         cudaGraphConditionalHandle cond, int use_cond, cudaStream_t st,
                         cudaEvent_t *ev) {
    // ev (optional): 2 * kRoundKernels events, recorded before/after each kernel
    const int sms = num_sms();
    int slot = 0;
    auto begin = [&] {
        if (ev) cudaEventRecord(ev[2 * slot], st);
    };
    auto end = [&] {
        if (ev) cudaEventRecord(ev[2 * slot + 1], st);
        ++slot;
    };
    const int issue_blocks = (int)std::min<int64_t>(ceil_div(a.nq, kIssueThreads), 8 * sms);
    begin();
    k_issue<<<issue_blocks, kIssueThreads, 0, st>>>(a);
    end();
    begin();
    k_bucket<<<1, kBucketThreads, 0, st>>>(a);
    end();
    const int scatter_blocks = (int)std::min<int64_t>(ceil_div(a.cap, 256), 8 * sms);
    begin();
    k_scatter<<<scatter_blocks, 256, 0, st>>>(a);
    end();
    begin();
    if (a.tc_min > 0) {
        if (a.rq)
            enqueue_scan_rq(a, st);
        else if (a.tc_stages)
            enqueue_scan_bulk(a, st);
        else
            enqueue_scan_tc(a, st);
    }
    end();
    begin();
    if (a.tc_min != 1)   // tc_min == 1 sends every group to the tensor cores
        k_scan<<<scan_blocks, kThreads, scan_smem, st>>>(a);
    end();
    const int merge_blocks = (int)std::min<int64_t>(ceil_div(a.nq * 32, kMergeThreads), 8 * sms);
    begin();
    k_merge<<<merge_blocks, kMergeThreads, 0, st>>>(a);
    end();
    begin();
    k_round_end<<<1, 1, 0, st>>>(a, cond, use_cond);
    end();
    return cudaGetLastError();
}

int scan_blocks_for(size_t smem) {
    int per_sm = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_scan, kThreads, smem);
    if (per_sm < 1) per_sm = 1;
    return per_sm * num_sms();
}

}  // namespace sieve
