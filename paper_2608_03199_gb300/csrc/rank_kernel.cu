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
    return round_up(b, 16);
}

__global__ void __launch_bounds__(kThreads) k_rank(const float *__restrict__ Q, int64_t nq,
                                                   const float *__restrict__ C, int64_t nlist,
                                                   int d, int nprobe, int32_t *__restrict__ order,
                                                   float *__restrict__ cscores) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int list_n[QT];
    float *Qst = reinterpret_cast<float *>(smem_raw);
    float *Cst = Qst + 2 * QT * LDX;
    float *Ss = Cst + 2 * RT * LDX;
    float *ls = Ss + QT * (RT + 1);
    int *lc = reinterpret_cast<int *>(ls + QT * nprobe);

    const int tid = threadIdx.x, tq = tid & 7, tr = tid >> 3;
    const unsigned lane = lane_id(), warp = tid >> 5;
    const int64_t q0 = (int64_t)blockIdx.x * QT;
    const int nqb = (int)(nq - q0 < QT ? nq - q0 : QT);
    const float *Qb = Q + q0 * d;
    if (tid < QT) list_n[tid] = 0;

    const int nch = (int)ceil_div(d, DK);
    const int64_t nsteps = ceil_div(nlist, RT) * nch;
    stage_rows<QT>(Qst, Qb, nqb, d, 0, 0);
    stage_rows<RT>(Cst, C, nlist, d, 0, 0);
    cp_async_commit();
    float acc[4][4];
    for (int64_t s = 0; s < nsteps; ++s) {
        const int64_t ct = s / nch;
        const int c = (int)(s % nch);
        if (s + 1 < nsteps) {
            const int64_t s1 = s + 1;
            const int b1 = (int)(s1 & 1);
            stage_rows<QT>(Qst + b1 * QT * LDX, Qb, nqb, d, 0, (int)(s1 % nch) * DK);
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
            for (int i = warp; i < nqb; i += kThreads / 32) {
                float *li_s = ls + i * nprobe;
                int *li_c = lc + i * nprobe;
                for (int half = 0; half < 2; ++half) {
                    const int64_t cid = ct * RT + half * 32 + lane;
                    const float sc = Ss[i * (RT + 1) + half * 32 + lane];
                    const int n = list_n[i];
                    bool cand = cid < nlist &&
                                (n < nprobe || ranks_before(sc, (int)cid, li_s[nprobe - 1],
                                                            li_c[nprobe - 1]));
                    unsigned bal = __ballot_sync(0xffffffffu, cand);
                    while (bal) {
                        const int src = __ffs(bal) - 1;
                        bal &= bal - 1;
                        const float bs = __shfl_sync(0xffffffffu, sc, src);
                        const int bc = __shfl_sync(0xffffffffu, (int)cid, src);
                        warp_list_insert(li_s, li_c, &list_n[i], nprobe, bs, bc);
                    }
                }
            }
        }
        __syncthreads();
    }
    for (int i = warp; i < nqb; i += kThreads / 32) {
        for (int j = lane; j < nprobe; j += 32) {
            order[(q0 + i) * nprobe + j] = lc[i * nprobe + j];
            if (cscores) cscores[(q0 + i) * nprobe + j] = ls[i * nprobe + j];
        }
    }
}

cudaError_t prepare_rank(int nprobe) {
    return cudaFuncSetAttribute(k_rank, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)rank_smem_bytes(nprobe));
}

cudaError_t enqueue_rank(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                         int nprobe, int32_t *order, float *cscores, cudaStream_t st) {
    if (nq == 0) return cudaSuccess;
    const int64_t blocks = ceil_div(nq, QT);
    k_rank<<<(unsigned)blocks, kThreads, rank_smem_bytes(nprobe), st>>>(Q, nq, C, nlist, d, nprobe,
                                                                       order, cscores);
    return cudaGetLastError();
}

}  // namespace sieve
