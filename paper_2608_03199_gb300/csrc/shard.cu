// shard.cu -- a query batch over several independent IVF indexes (the
// public-100M layout of Sec. 6.1: coarse shards, each with its own IVF index,
// searched with its own ranking and stopping): the global top-k merge of the
// shards' results, by (score desc, id asc).
#include "search.cuh"

namespace sieve {

constexpr int kShardMergeThreads = 256;

// one warp per query; the running top-k (k <= 64) in two registers per lane,
// each shard's sorted list inserted in order until its entries rank too low
__global__ void __launch_bounds__(kShardMergeThreads) k_merge_shards(
    int nshards, int64_t nq, int k, const long long *__restrict__ ids, const float *__restrict__ sc,
    const int *__restrict__ cnt, const int *__restrict__ pr, long long *__restrict__ out_ids,
    float *__restrict__ out_sc, int *__restrict__ out_cnt, int *__restrict__ out_pr,
    int *__restrict__ shard_probes) {
    const unsigned lane = lane_id();
    const int64_t gw = ((int64_t)blockIdx.x * kShardMergeThreads + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * kShardMergeThreads) >> 5;
    const float ninf = -__int_as_float(0x7f800000);
    for (int64_t q = gw; q < nq; q += nw) {
        int n = 0, probes = 0;
        float r0s = ninf, r1s = ninf;
        long long r0i = -1, r1i = -1;
        for (int s = 0; s < nshards; ++s) {
            const int64_t row = (int64_t)s * nq + q;
            const int c = cnt[row];
            probes += pr[row];
            if (shard_probes && lane == 0) shard_probes[q * nshards + s] = pr[row];
            for (int j = 0; j < c; ++j) {
                const float v = sc[row * k + j];
                const long long id = ids[row * k + j];
                const bool b0 = (int)lane < n && ranks_before(r0s, r0i, v, id);
                const bool b1 = (int)lane + 32 < n && ranks_before(r1s, r1i, v, id);
                const int pos = __popc(__ballot_sync(0xffffffffu, b0)) +
                                __popc(__ballot_sync(0xffffffffu, b1));
                if (pos >= k) break;   // the rest of this sorted list ranks lower
                float u0s = __shfl_up_sync(0xffffffffu, r0s, 1);
                long long u0i = __shfl_up_sync(0xffffffffu, r0i, 1);
                float u1s = __shfl_up_sync(0xffffffffu, r1s, 1);
                long long u1i = __shfl_up_sync(0xffffffffu, r1i, 1);
                const float w31s = __shfl_sync(0xffffffffu, r0s, 31);
                const long long w31i = __shfl_sync(0xffffffffu, r0i, 31);
                if (lane == 0) { u1s = w31s; u1i = w31i; }
                const int j0 = lane, j1 = lane + 32;
                if (j0 == pos) { r0s = v; r0i = id; }
                else if (j0 > pos) { r0s = u0s; r0i = u0i; }
                if (j1 == pos) { r1s = v; r1i = id; }
                else if (j1 > pos) { r1s = u1s; r1i = u1i; }
                n = n < k ? n + 1 : k;
            }
        }
        const int64_t ob = q * k;
        if ((int)lane < k) {
            out_sc[ob + lane] = (int)lane < n ? r0s : ninf;
            out_ids[ob + lane] = (int)lane < n ? r0i : -1;
        }
        if ((int)lane + 32 < k) {
            out_sc[ob + lane + 32] = (int)lane + 32 < n ? r1s : ninf;
            out_ids[ob + lane + 32] = (int)lane + 32 < n ? r1i : -1;
        }
        if (lane == 0) {
            out_cnt[q] = n;
            out_pr[q] = probes;
        }
    }
}

cudaError_t launch_merge_shards(int nshards, int64_t nq, int k, const long long *ids, const float *sc,
                                const int *cnt, const int *pr, long long *out_ids, float *out_sc,
                                int *out_cnt, int *out_pr, int *shard_probes, cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    const int64_t blocks = std::min<int64_t>(ceil_div(nq * 32, kShardMergeThreads), 8 * (int64_t)num_sms());
    k_merge_shards<<<(unsigned)blocks, kShardMergeThreads, 0, st>>>(
        nshards, nq, k, ids, sc, cnt, pr, out_ids, out_sc, out_cnt, out_pr, shard_probes);
    return cudaGetLastError();
}

}  // namespace sieve
