// calibrate.cu -- in-call window calibration (Appendix A, Algorithm 3): the
// device steps around two searches.
//
//   k_gather_rows / k_gather_ids   copy the sampled (or the remaining) queries
//   k_complement                   the row indices of Q not in the sample
//   k_calib_hist                   RequiredWindowHistogram: a sampled query's
//                                  neighbour found at rank j needs a window of
//                                  1 + the longest run of empty ranks before j
//   k_calib_pick                   the smallest W < nprobe whose loss
//                                  1 - (H[1] + .. + H[W]) / Z is below eps
//   k_scatter_results              search outputs back to their batch rows
#include "search.cuh"

namespace sieve {

// out[i][*] = src[idx[i]][*] for rows of `width` floats (width a multiple of 4)
__global__ void k_gather_rows(const float *__restrict__ src, int width, const int64_t *__restrict__ idx,
                              int64_t n, float *__restrict__ out) {
    const int v4 = width / 4;
    const int64_t total = n * v4;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = u / v4;
        const int c = (int)(u % v4);
        reinterpret_cast<float4 *>(out + i * width)[c] =
            reinterpret_cast<const float4 *>(src + idx[i] * width)[c];
    }
}

__global__ void k_gather_ids(const int64_t *__restrict__ src, const int64_t *__restrict__ idx,
                             int64_t n, int64_t *__restrict__ out) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        out[i] = src[idx[i]];
}

// rest[i] = the i-th row index of [0, nq) missing from the sorted, distinct
// sample: the smallest x with x + 1 - #{sample <= x} = i + 1
__global__ void k_complement(const int64_t *__restrict__ sample, int64_t ns, int64_t nq,
                             int64_t *__restrict__ rest) {
    const int64_t nr = nq - ns;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nr;
         i += (int64_t)gridDim.x * blockDim.x) {
        int64_t lo = i, hi = i + ns;   // the answer lies in [i, i + ns]
        while (lo < hi) {
            const int64_t x = (lo + hi) >> 1;
            int64_t a = 0, b = ns;     // #{sample <= x}
            while (a < b) {
                const int64_t m = (a + b) >> 1;
                if (sample[m] <= x) a = m + 1; else b = m;
            }
            if (x + 1 - a >= i + 1) hi = x; else lo = x + 1;
        }
        rest[i] = lo;
    }
}

// one thread per sampled query: walk its ranks in order, keeping the longest
// run of empty ranks so far; each kept result found at rank j adds one to
// H[1 + that run before j]; Z sums the kept results
__global__ void k_calib_hist(const unsigned *__restrict__ hit_bits, int words,
                             const int *__restrict__ out_rank, const int *__restrict__ count,
                             int64_t ns, int k, int nprobe, unsigned long long *__restrict__ hist,
                             unsigned long long *__restrict__ Z) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < ns;
         i += (int64_t)gridDim.x * blockDim.x) {
        const unsigned *hb = hit_bits + i * words;
        const int *rk = out_rank + i * k;
        const int c = count[i];
        int run = 0, longest = 0, left = c;
        for (int j = 1; j <= nprobe && left > 0; ++j) {
            const bool hit = (hb[(j - 1) >> 5] >> ((j - 1) & 31)) & 1u;
            if (hit) {
                int here = 0;
                for (int e = 0; e < c; ++e) here += rk[e] == j;
                if (here) {
                    atomicAdd(&hist[1 + longest], (unsigned long long)here);
                    left -= here;
                }
            }
            run = hit ? 0 : run + 1;
            if (run > longest) longest = run;
        }
        if (c) atomicAdd(Z, (unsigned long long)c);
    }
}

// W* (Algorithm 3): the fallback when no sampled query kept a result
__global__ void k_calib_pick(const unsigned long long *__restrict__ hist,
                             const unsigned long long *__restrict__ Z, int nprobe, double eps,
                             int fallback, int *__restrict__ W_out) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    const unsigned long long z = *Z;
    int w_star = nprobe;
    if (z == 0) {
        w_star = fallback;
    } else {
        unsigned long long retained = 0;
        for (int w = 1; w < nprobe; ++w) {
            retained += hist[w];
            const double loss = 1.0 - (double)retained / (double)z;
            if (loss < eps) {
                w_star = w;
                break;
            }
        }
    }
    *W_out = w_star;
}

// row i of the search outputs goes to batch row idx[i]
__global__ void k_scatter_results(const int64_t *__restrict__ idx, int64_t n, int k,
                                  const long long *__restrict__ ids, const float *__restrict__ sc,
                                  const int *__restrict__ cnt, const int *__restrict__ pr,
                                  long long *__restrict__ out_ids, float *__restrict__ out_sc,
                                  int *__restrict__ out_cnt, int *__restrict__ out_pr) {
    const int64_t total = n * k;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = u / k;
        const int e = (int)(u % k);
        const int64_t to = idx[i];
        out_ids[to * k + e] = ids[u];
        out_sc[to * k + e] = sc[u];
        if (e == 0) {
            out_cnt[to] = cnt[i];
            out_pr[to] = pr[i];
        }
    }
}

// the sample must be strictly increasing row indices of [0, nq)
__global__ void k_check_sample(const int64_t *__restrict__ sample, int64_t ns, int64_t nq,
                               int *__restrict__ bad) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < ns;
         i += (int64_t)gridDim.x * blockDim.x)
        if (sample[i] < 0 || sample[i] >= nq || (i > 0 && sample[i] <= sample[i - 1])) *bad = 1;
}

static int grid_for(int64_t n, int threads) {
    const int64_t b = ceil_div(n > 0 ? n : 1, threads);
    const int64_t cap = 8 * (int64_t)num_sms();
    return (int)(b < cap ? b : cap);
}

cudaError_t calib_gather(const float *Q, const int64_t *qids, int d, const int64_t *idx, int64_t n,
                         float *Qo, int64_t *qo, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_gather_rows<<<grid_for(n * (d / 4), 256), 256, 0, st>>>(Q, d, idx, n, Qo);
    if (qids) k_gather_ids<<<grid_for(n, 256), 256, 0, st>>>(qids, idx, n, qo);
    return cudaGetLastError();
}

cudaError_t calib_check_sample(const int64_t *sample, int64_t ns, int64_t nq, int *bad,
                               cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(bad, 0, sizeof(int), st);
    if (e != cudaSuccess || ns <= 0) return e;
    k_check_sample<<<grid_for(ns, 256), 256, 0, st>>>(sample, ns, nq, bad);
    return cudaGetLastError();
}

cudaError_t calib_complement(const int64_t *sample, int64_t ns, int64_t nq, int64_t *rest,
                             cudaStream_t st) {
    if (nq - ns <= 0) return cudaSuccess;
    k_complement<<<grid_for(nq - ns, 256), 256, 0, st>>>(sample, ns, nq, rest);
    return cudaGetLastError();
}

cudaError_t calib_pick(const unsigned *hit_bits, int words, const int *out_rank, const int *count,
                       int64_t ns, int k, int nprobe, double eps, int fallback,
                       unsigned long long *hist, unsigned long long *Z, int *W_out,
                       cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(hist, 0, sizeof(unsigned long long) * (nprobe + 1), st);
    if (e == cudaSuccess) e = cudaMemsetAsync(Z, 0, sizeof(unsigned long long), st);
    if (e != cudaSuccess) return e;
    if (ns > 0)
        k_calib_hist<<<grid_for(ns, 128), 128, 0, st>>>(hit_bits, words, out_rank, count, ns, k,
                                                      nprobe, hist, Z);
    k_calib_pick<<<1, 32, 0, st>>>(hist, Z, nprobe, eps, fallback, W_out);
    return cudaGetLastError();
}

cudaError_t calib_scatter(const int64_t *idx, int64_t n, int k, const long long *ids, const float *sc,
                          const int *cnt, const int *pr, long long *out_ids, float *out_sc,
                          int *out_cnt, int *out_pr, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_scatter_results<<<grid_for(n * k, 256), 256, 0, st>>>(idx, n, k, ids, sc, cnt, pr, out_ids,
                                                           out_sc, out_cnt, out_pr);
    return cudaGetLastError();
}

}  // namespace sieve
