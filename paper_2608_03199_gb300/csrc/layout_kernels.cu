// layout_kernels.cu -- partition-contiguous storage of an IVF index (Sec. 2.3):
// a counting sort of the rows by partition, rows of one partition kept in
// increasing row order.
//
//   k_layout_hist   per-partition counts (and a flag for assign out of range)
//   k_layout_scan   one block: exclusive prefix sums -> list_offsets, cursors
//   k_layout_place  each row claims a slot in its partition (atomic cursor)
//   k_layout_order  one block per partition: bitonic sort of the claimed row
//                   indices (shared memory, or a padded global scratch area
//                   for partitions above kSmemSortMax rows)
//   k_layout_copy   one warp per sorted row: gather the vector
#include "search.cuh"

namespace sieve {

constexpr int kSortThreads = 1024;
constexpr int64_t kSmemSortMax = 8192;   // int64 keys sorted in shared memory

size_t layout_workspace_bytes(int64_t n, int64_t nlist) {
    // counts/cursors [nlist] u64, flag, and a 2n-slot scratch for large partitions
    return (size_t)round_up((nlist + 1) * 8, 256) + 256 + (size_t)round_up(2 * n * 8, 256);
}

__global__ void k_layout_hist(const int32_t *assign, int64_t n, int64_t nlist,
                              unsigned long long *counts, int *bad) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        int32_t p = assign[i];
        if (p < 0 || p >= nlist) {
            atomicExch(bad, 1);
            continue;
        }
        atomicAdd(&counts[p], 1ull);
    }
}

__global__ void __launch_bounds__(1024) k_layout_scan(unsigned long long *counts, int64_t nlist,
                                                      int64_t *offsets) {
    __shared__ unsigned long long warp_tot[32];
    const int per = (int)ceil_div(nlist, 1024);
    const int64_t p0 = (int64_t)threadIdx.x * per;
    unsigned long long mine = 0;
    for (int64_t p = p0; p < p0 + per && p < nlist; ++p) mine += counts[p];
    const unsigned lane = lane_id(), warp = threadIdx.x >> 5;
    unsigned long long x = mine;
    for (int o = 1; o < 32; o <<= 1) {
        unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= (unsigned)o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        unsigned long long w = warp_tot[lane];
        for (int o = 1; o < 32; o <<= 1) {
            unsigned long long y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= (unsigned)o) w += y;
        }
        warp_tot[lane] = w;
    }
    __syncthreads();
    unsigned long long run = (warp > 0 ? warp_tot[warp - 1] : 0) + x - mine;
    for (int64_t p = p0; p < p0 + per && p < nlist; ++p) {
        unsigned long long c = counts[p];
        offsets[p] = (int64_t)run;
        counts[p] = run;   // becomes the placement cursor
        run += c;
    }
    if (threadIdx.x == 1023) offsets[nlist] = (int64_t)run;
}

__global__ void k_layout_place(const int32_t *assign, int64_t n, int64_t nlist,
                               unsigned long long *cursor, int64_t *ids_sorted) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        int32_t p = assign[i];
        if (p < 0 || p >= nlist) continue;
        unsigned long long pos = atomicAdd(&cursor[p], 1ull);
        ids_sorted[pos] = i;
    }
}

// ascending bitonic sort of a[0..L), L a power of two, by one thread block
__device__ void block_bitonic_sort(int64_t *a, int64_t L) {
    for (int64_t size = 2; size <= L; size <<= 1) {
        for (int64_t stride = size >> 1; stride > 0; stride >>= 1) {
            for (int64_t i = threadIdx.x; i < L / 2; i += blockDim.x) {
                int64_t lo = 2 * i - (i & (stride - 1));
                int64_t hi = lo + stride;
                bool up = (lo & size) == 0;
                int64_t x = a[lo], y = a[hi];
                if ((x > y) == up) {
                    a[lo] = y;
                    a[hi] = x;
                }
            }
            __syncthreads();
        }
    }
}

__global__ void __launch_bounds__(kSortThreads) k_layout_order(const int64_t *offsets,
                                                               int64_t *ids_sorted,
                                                               int64_t *scratch) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int64_t p = blockIdx.x;
    const int64_t b = offsets[p], m = offsets[p + 1] - b;
    if (m <= 1) return;
    int64_t L = 1;
    while (L < m) L <<= 1;
    int64_t *a = (L <= kSmemSortMax) ? reinterpret_cast<int64_t *>(smem_raw) : scratch + 2 * b;
    for (int64_t i = threadIdx.x; i < L; i += blockDim.x)
        a[i] = i < m ? ids_sorted[b + i] : INT64_MAX;
    __syncthreads();
    block_bitonic_sort(a, L);
    for (int64_t i = threadIdx.x; i < m; i += blockDim.x) ids_sorted[b + i] = a[i];
}

__global__ void k_layout_copy(const float *X, int64_t n, int d, const int64_t *ids_sorted,
                              float *X_sorted, const int *bad) {
    if (*bad) return;   // some rows were not placed: ids_sorted is incomplete
    const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const unsigned lane = lane_id();
    const int nv = d / 4;
    for (int64_t j = w; j < n; j += nw) {
        const float4 *src = reinterpret_cast<const float4 *>(X + ids_sorted[j] * d);
        float4 *dst = reinterpret_cast<float4 *>(X_sorted + j * d);
        for (int v = lane; v < nv; v += 32) dst[v] = src[v];
    }
}

cudaError_t launch_layout(const float *X, const int32_t *assign, int64_t n, int d, int64_t nlist,
                          float *X_sorted, int64_t *ids_sorted, int64_t *list_offsets, void *ws,
                          int *bad_flag_host, cudaStream_t st) {
    unsigned char *w = static_cast<unsigned char *>(ws);
    unsigned long long *counts = reinterpret_cast<unsigned long long *>(w);
    int *bad = reinterpret_cast<int *>(w + round_up((nlist + 1) * 8, 256));
    int64_t *scratch = reinterpret_cast<int64_t *>(w + round_up((nlist + 1) * 8, 256) + 256);
    cudaError_t e;
    if ((e = cudaMemsetAsync(counts, 0, (size_t)(nlist + 1) * 8, st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(bad, 0, sizeof(int), st)) != cudaSuccess) return e;
    const int sms = num_sms();
    int blocks = (int)std::min<int64_t>(ceil_div(n > 0 ? n : 1, 256), 16 * sms);
    k_layout_hist<<<blocks, 256, 0, st>>>(assign, n, nlist, counts, bad);
    k_layout_scan<<<1, 1024, 0, st>>>(counts, nlist, list_offsets);
    k_layout_place<<<blocks, 256, 0, st>>>(assign, n, nlist, counts, ids_sorted);
    const size_t smem = kSmemSortMax * sizeof(int64_t);
    if ((e = cudaFuncSetAttribute(k_layout_order, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)smem)) != cudaSuccess)
        return e;
    if (nlist > 0) k_layout_order<<<(unsigned)nlist, kSortThreads, smem, st>>>(list_offsets, ids_sorted, scratch);
    int cblocks = (int)std::min<int64_t>(ceil_div(n > 0 ? n : 1, 8), 16 * sms);
    k_layout_copy<<<cblocks, 256, 0, st>>>(X, n, d, ids_sorted, X_sorted, bad);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = cudaMemcpyAsync(bad_flag_host, bad, sizeof(int), cudaMemcpyDeviceToHost, st)) !=
        cudaSuccess)
        return e;
    return cudaStreamSynchronize(st);
}

}  // namespace sieve
