// rank_kernel.cu -- centroid ranking with a fused per-query top-nprobe
// (Sec. 2.3, Sec. 4.1: P_i = the nprobe centroids closest to q_i, closest
// first; for unit vectors the closest by cosine has the largest inner
// product; equal scores rank the lower centroid id first).
//
// One block owns QT queries and streams every centroid through shared memory
// in tiles of RT, staging QT x DK query columns and RT x DK centroid columns
// per pipeline step (cp.async, double buffered).  After each centroid tile
// the scores go to shared memory and one warp per query merges the tile into
// that query's sorted top-nprobe list (kept in shared memory; a score enters
// only if it ranks before the current last entry).  The score matrix is never
// written to global memory.
#include "search.cuh"

namespace sieve {

size_t rank_smem_bytes(int nprobe) {
    size_t b = 0;
    b += 2ull * QT * LDX * sizeof(float);        // query chunks
    b += 2ull * RT * LDX * sizeof(float);        // centroid chunks
    b += (size_t)QT * (RT + 1) * sizeof(float);  // tile scores
    b += (size_t)QT * nprobe * sizeof(float);    // list scores
    b += (size_t)QT * nprobe * sizeof(int);      // list ids
    b += (size_t)(kThreads / 32) * RT * 8;       // per-warp sorted tile
    b += (size_t)(kThreads / 32) * nprobe * 8;   // per-warp merge output
    return round_up(b, 16);
}

// Sort the 64 entries of a warp (entry h*32 + lane in slot h) so that entry 0
// ranks first (score desc, id asc): a bitonic network, shuffles within a half,
// in-register exchange across the halves.
__device__ __forceinline__ void warp_sort64(float (&s)[2], int (&c)[2]) {
    const unsigned lane = lane_id();
    for (int k = 2; k <= 64; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
            if (j == 32) {
                // pair (lane, lane + 32); k == 64 here, so the block sorts "first first"
                if (!ranks_before(s[0], c[0], s[1], c[1])) {
                    float ts = s[0]; s[0] = s[1]; s[1] = ts;
                    int tc = c[0]; c[0] = c[1]; c[1] = tc;
                }
            } else {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int e = h * 32 + (int)lane;
                    const float ps = __shfl_xor_sync(0xffffffffu, s[h], j);
                    const int pc = __shfl_xor_sync(0xffffffffu, c[h], j);
                    const bool up = (e & k) == 0;       // this block sorts first-ranked first
                    const bool lower = (e & j) == 0;    // the lower index of the pair
                    const bool mine_first = ranks_before(s[h], c[h], ps, pc);
                    if (mine_first != (lower == up)) {
                        s[h] = ps;
                        c[h] = pc;
                    }
                }
            }
        }
    }
}

// Merge the sorted list L (n entries, capacity cap) with the sorted tile T
// (its first m entries) and keep the first cap: merge-path co-ranks, one
// output position per lane step.  O is per-warp scratch of cap entries.
__device__ __forceinline__ void warp_merge_list(float *Ls, int *Lc, int *n_ptr, int cap,
                                                const float *Ts, const int *Tc, int m,
                                                float *Os, int *Oc) {
    const unsigned lane = lane_id();
    const int n = *n_ptr;
    const int total = n + m < cap ? n + m : cap;
    for (int j = lane; j < total; j += 32) {
        int lo = j - m > 0 ? j - m : 0;
        int hi = j < n ? j : n;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (ranks_before(Ls[mid], Lc[mid], Ts[j - mid - 1], Tc[j - mid - 1]))
                lo = mid + 1;
            else
                hi = mid;
        }
        const int i = lo;
        const bool take_l = i < n && (j - i >= m || ranks_before(Ls[i], Lc[i], Ts[j - i], Tc[j - i]));
        Os[j] = take_l ? Ls[i] : Ts[j - i];
        Oc[j] = take_l ? Lc[i] : Tc[j - i];
    }
    __syncwarp();
    for (int j = lane; j < total; j += 32) {
        Ls[j] = Os[j];
        Lc[j] = Oc[j];
    }
    if (lane == 0) *n_ptr = total;
    __syncwarp();
}

// QT query rows of Q given by row index (rows >= nrows and columns >= d are
// zero-filled): DK columns from c0 into Xs[QT][LDX], like stage_rows
__device__ __forceinline__ void stage_query_rows(float *Xs, const float *__restrict__ Q,
                                                 const int64_t *qrow, int nrows, int d, int c0) {
    constexpr int kVec = DK / 4;
    for (int idx = threadIdx.x; idx < QT * kVec; idx += kThreads) {
        const int r = idx / kVec, v = idx % kVec;
        const int col = c0 + 4 * v;
        const bool ok = r < nrows && col < d;
        const float *src = ok ? Q + qrow[r] * (int64_t)d + col : Q;
        cp_async16(Xs + r * LDX + 4 * v, src, ok ? 16 : 0);
    }
}

// qlist (nullable): rank only the queries qlist[0 .. *qlist_n - 1] (rows of Q
// and of order/cscores); block b takes list entries b*QT .. b*QT+QT-1
__global__ void __launch_bounds__(kThreads) k_rank(const float *__restrict__ Q, int64_t nq,
                                                   const float *__restrict__ C, int64_t nlist,
                                                   int d, int nprobe, int32_t *__restrict__ order,
                                                   float *__restrict__ cscores,
                                                   const int *__restrict__ qlist,
                                                   const int *__restrict__ qlist_n) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int list_n[QT];
    float *Qst = reinterpret_cast<float *>(smem_raw);
    float *Cst = Qst + 2 * QT * LDX;
    float *Ss = Cst + 2 * RT * LDX;
    float *ls = Ss + QT * (RT + 1);
    int *lc = reinterpret_cast<int *>(ls + QT * nprobe);
    float *ts_w = reinterpret_cast<float *>(lc + QT * nprobe) + (threadIdx.x >> 5) * (2 * RT);
    int *tc_w = reinterpret_cast<int *>(ts_w + RT);
    float *os_w = reinterpret_cast<float *>(lc + QT * nprobe) + (kThreads / 32) * 2 * RT +
                  (threadIdx.x >> 5) * (2 * nprobe);
    int *oc_w = reinterpret_cast<int *>(os_w + nprobe);

    __shared__ int64_t qrow[QT];   // the block's queries (rows of Q and of order)
    const int tid = threadIdx.x, tq = tid & 7, tr = tid >> 3;
    const unsigned lane = lane_id(), warp = tid >> 5;
    const int64_t q0 = (int64_t)blockIdx.x * QT;
    const int64_t nsel = qlist ? (int64_t)*qlist_n : nq;
    if (q0 >= nsel) return;
    const int nqb = (int)(nsel - q0 < QT ? nsel - q0 : QT);
    if (tid < QT) {
        list_n[tid] = 0;
        qrow[tid] = tid < nqb ? (qlist ? (int64_t)qlist[q0 + tid] : q0 + tid) : 0;
    }
    __syncthreads();

    const int nch = (int)ceil_div(d, DK);
    const int64_t nsteps = ceil_div(nlist, RT) * nch;
    stage_query_rows(Qst, Q, qrow, nqb, d, 0);
    stage_rows<RT>(Cst, C, nlist, d, 0, 0);
    cp_async_commit();
    float acc[4][4];
    for (int64_t s = 0; s < nsteps; ++s) {
        const int64_t ct = s / nch;
        const int c = (int)(s % nch);
        if (s + 1 < nsteps) {
            const int64_t s1 = s + 1;
            const int b1 = (int)(s1 & 1);
            stage_query_rows(Qst + b1 * QT * LDX, Q, qrow, nqb, d, (int)(s1 % nch) * DK);
            stage_rows<RT>(Cst + b1 * RT * LDX, C, nlist, d, (s1 / nch) * RT, (int)(s1 % nch) * DK);
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
        const int b = (int)(s & 1);
        contract_chunk(acc, Qst + b * QT * LDX, LDX, 0, Cst + b * RT * LDX, tq, tr);
        if (c == nch - 1) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) Ss[(tq + 8 * i) * (RT + 1) + tr + 16 * j] = acc[i][j];
            __syncthreads();
            // merge the tile into each query's sorted top-nprobe list: entries
            // that rank before the list's last entry are candidates; a few are
            // inserted one by one, more are sorted and merged in one pass
            for (int i = warp; i < nqb; i += kThreads / 32) {
                float *li_s = ls + i * nprobe;
                int *li_c = lc + i * nprobe;
                const int n = list_n[i];
                float sv[2];
                int cv[2];
                bool cand[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int64_t cid = ct * RT + h * 32 + lane;
                    sv[h] = cid < nlist ? Ss[i * (RT + 1) + h * 32 + lane] : -__int_as_float(0x7f800000);
                    cv[h] = cid < nlist ? (int)cid : INT32_MAX;
                    cand[h] = cid < nlist &&
                              (n < nprobe || ranks_before(sv[h], cv[h], li_s[nprobe - 1], li_c[nprobe - 1]));
                }
                const unsigned b0 = __ballot_sync(0xffffffffu, cand[0]);
                const unsigned b1 = __ballot_sync(0xffffffffu, cand[1]);
                const int m = __popc(b0) + __popc(b1);
                if (m == 0) continue;
                if (m <= 4) {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        unsigned bal = h ? b1 : b0;
                        while (bal) {
                            const int src = __ffs(bal) - 1;
                            bal &= bal - 1;
                            const float bs = __shfl_sync(0xffffffffu, sv[h], src);
                            const int bc = __shfl_sync(0xffffffffu, cv[h], src);
                            warp_list_insert(li_s, li_c, &list_n[i], nprobe, bs, bc);
                        }
                    }
                } else {
                    // candidates form a prefix of the sorted tile
                    warp_sort64(sv, cv);
                    ts_w[lane] = sv[0];
                    tc_w[lane] = cv[0];
                    ts_w[lane + 32] = sv[1];
                    tc_w[lane + 32] = cv[1];
                    __syncwarp();
                    warp_merge_list(li_s, li_c, &list_n[i], nprobe, ts_w, tc_w, m, os_w, oc_w);
                }
            }
        }
        __syncthreads();
    }
    for (int i = warp; i < nqb; i += kThreads / 32) {
        for (int j = lane; j < nprobe; j += 32) {
            order[qrow[i] * nprobe + j] = lc[i * nprobe + j];
            if (cscores) cscores[qrow[i] * nprobe + j] = ls[i * nprobe + j];
        }
    }
}

cudaError_t prepare_rank(int nprobe) {
    return cudaFuncSetAttribute(k_rank, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)rank_smem_bytes(nprobe));
}

cudaError_t enqueue_rank(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                         int nprobe, int32_t *order, float *cscores, cudaStream_t st,
                         const int *qlist, const int *qlist_n) {
    if (nq == 0) return cudaSuccess;
    const int64_t blocks = ceil_div(nq, QT);
    k_rank<<<(unsigned)blocks, kThreads, rank_smem_bytes(nprobe), st>>>(Q, nq, C, nlist, d, nprobe,
                                                                       order, cscores, qlist, qlist_n);
    return cudaGetLastError();
}

}  // namespace sieve
