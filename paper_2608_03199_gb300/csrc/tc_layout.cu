// tc_layout.cu -- the tensor-core layout of an index: partition rows and
// centroids stored already split for the fp16 contraction, in the exact
// byte order of the shared-memory operand tiles, so the scan streams them
// with bulk copies instead of converting on every pass.
//
// A matrix (one partition's rows, or all centroids) is cut into blocks of
// kTcRows = 128 rows; rows past the end of the matrix are zero.  For each
// K-block kb of 64 elements a block stores 16 KB of hi fp16 then 16 KB of lo
// fp16 (hi = fp16(256 x), lo = fp16(256 x - hi), as in tc_pipeline.cuh),
// each a 128-row x 128-byte tile whose 16-byte chunk c of row r sits at
// chunk c ^ (r & 7).  Block b, K-block kb of the matrix starts at byte
// (b * nkb + kb) * 32768.  Partition p owns blocks blk_off[p] .. blk_off[p+1]-1.
// The row layout ends with one fp32 per block, the largest Euclidean norm of
// its rows: the screening scan bounds the error of its one-product scores
// with it.
#include <cuda_fp16.h>

#include "search.cuh"

namespace sieve {

__global__ void __launch_bounds__(1024) k_tc_block_scan(const int64_t *off, int64_t nparts,
                                                        int64_t *blk_off) {
    __shared__ long long warp_tot[32];
    const int per = (int)ceil_div(nparts, 1024);
    const int64_t p0 = (int64_t)threadIdx.x * per;
    long long mine = 0;
    for (int64_t p = p0; p < p0 + per && p < nparts; ++p) mine += ceil_div(off[p + 1] - off[p], kTcRows);
    const unsigned lane = lane_id(), warp = threadIdx.x >> 5;
    long long x = mine;
    for (int o = 1; o < 32; o <<= 1) {
        long long y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= (unsigned)o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        long long w = warp_tot[lane];
        for (int o = 1; o < 32; o <<= 1) {
            long long y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= (unsigned)o) w += y;
        }
        warp_tot[lane] = w;
    }
    __syncthreads();
    long long run = (warp > 0 ? warp_tot[warp - 1] : 0) + x - mine;
    for (int64_t p = p0; p < p0 + per && p < nparts; ++p) {
        blk_off[p] = run;
        run += ceil_div(off[p + 1] - off[p], kTcRows);
    }
    if (threadIdx.x == 1023) blk_off[nparts] = run;
}

__device__ __forceinline__ void split2h(float a, float b, uint32_t &hi, uint32_t &lo) {
    const float2 f = make_float2(a * 256.f, b * 256.f);
    const __half2 h = __float22half2_rn(f);
    const float2 back = __half22float2(h);
    const __half2 l = __float22half2_rn(make_float2(f.x - back.x, f.y - back.y));
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

// one thread per (block, K-block, row, 16-byte chunk); off == nullptr means a
// single matrix of nrows rows (the centroids), blk_off unused
__global__ void k_tc_fill(const float *X, const int64_t *off, int64_t nparts, int64_t nrows,
                          const int64_t *blk_off, int d, int nkb, unsigned char *out) {
    const int64_t nblocks = off ? blk_off[nparts] : ceil_div(nrows, kTcRows);
    const int64_t total = nblocks * nkb * kTcRows * 8;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(u & 7);
        const int r = (int)((u >> 3) & (kTcRows - 1));
        const int64_t bk = u >> 10;             // block * nkb + kb
        const int kb = (int)(bk % nkb);
        const int64_t blk = bk / nkb;
        int64_t row, end;
        if (off) {
            int64_t lo_p = 0, hi_p = nparts;    // partition: blk_off[p] <= blk < blk_off[p + 1]
            while (hi_p - lo_p > 1) {
                const int64_t mid = (lo_p + hi_p) >> 1;
                if (blk_off[mid] <= blk) lo_p = mid; else hi_p = mid;
            }
            row = off[lo_p] + (blk - blk_off[lo_p]) * kTcRows + r;
            end = off[lo_p + 1];
        } else {
            row = blk * kTcRows + r;
            end = nrows;
        }
        const bool valid = row < end;
        const int col = kb * 64 + c * 8;
        float4 x0 = make_float4(0.f, 0.f, 0.f, 0.f), x1 = x0;
        if (valid && col < d) x0 = *reinterpret_cast<const float4 *>(X + row * d + col);
        if (valid && col + 4 < d) x1 = *reinterpret_cast<const float4 *>(X + row * d + col + 4);
        uint4 h, l;
        split2h(x0.x, x0.y, h.x, l.x);
        split2h(x0.z, x0.w, h.y, l.y);
        split2h(x1.x, x1.y, h.z, l.z);
        split2h(x1.z, x1.w, h.w, l.w);
        unsigned char *dst = out + bk * kTcBlockBytes + (int64_t)r * 128 + ((c ^ (r & 7)) << 4);
        *reinterpret_cast<uint4 *>(dst) = h;
        *reinterpret_cast<uint4 *>(dst + kTcBlockBytes / 2) = l;
    }
}

// a warp per block of partition rows: the largest norm of the block's rows,
// stored after the blocks (fp32 sums of squares; the screening bound leaves
// room for their rounding)
__global__ void k_tc_norms(const float *X, const int64_t *off, int64_t nparts, const int64_t *blk_off,
                           int d, int nkb, unsigned char *out) {
    const int64_t nblocks = blk_off[nparts];
    float *norms = reinterpret_cast<float *>(out + nblocks * nkb * kTcBlockBytes);
    const int lane = (int)lane_id();
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t blk = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; blk < nblocks; blk += warps) {
        int64_t lo_p = 0, hi_p = nparts;    // partition: blk_off[p] <= blk < blk_off[p + 1]
        while (hi_p - lo_p > 1) {
            const int64_t mid = (lo_p + hi_p) >> 1;
            if (blk_off[mid] <= blk) lo_p = mid; else hi_p = mid;
        }
        const int64_t r0 = off[lo_p] + (blk - blk_off[lo_p]) * kTcRows;
        const int64_t r1 = r0 + kTcRows < off[lo_p + 1] ? r0 + kTcRows : off[lo_p + 1];
        float best = 0.f;
        for (int64_t r = r0; r < r1; ++r) {
            float ss = 0.f;
            for (int c = 4 * lane; c < d; c += 128) {
                const float4 x = __ldg(reinterpret_cast<const float4 *>(X + r * d + c));
                ss = fmaf(x.x, x.x, fmaf(x.y, x.y, fmaf(x.z, x.z, fmaf(x.w, x.w, ss))));
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
            best = fmaxf(best, sqrtf(ss));
        }
        if (lane == 0) norms[blk] = best;
    }
}

int tc_nkb(int d) { return (int)ceil_div(d, 64); }

size_t tc_norms_bytes(int64_t nblocks) { return (size_t)round_up(nblocks * 4, 256); }

cudaError_t launch_tc_block_scan(const int64_t *off, int64_t nparts, int64_t *blk_off, cudaStream_t st) {
    k_tc_block_scan<<<1, 1024, 0, st>>>(off, nparts, blk_off);
    return cudaGetLastError();
}

cudaError_t launch_tc_layout_rows(const float *X, const int64_t *off, int64_t nparts, int d,
                                  int64_t *blk_off, unsigned char *out, cudaStream_t st) {
    k_tc_block_scan<<<1, 1024, 0, st>>>(off, nparts, blk_off);
    k_tc_fill<<<16 * num_sms(), 256, 0, st>>>(X, off, nparts, 0, blk_off, d, tc_nkb(d), out);
    k_tc_norms<<<8 * num_sms(), 256, 0, st>>>(X, off, nparts, blk_off, d, tc_nkb(d), out);
    return cudaGetLastError();
}

cudaError_t launch_tc_layout_matrix(const float *X, int64_t nrows, int d, unsigned char *out,
                                    cudaStream_t st) {
    k_tc_fill<<<16 * num_sms(), 256, 0, st>>>(X, nullptr, 1, nrows, nullptr, d, tc_nkb(d), out);
    return cudaGetLastError();
}

}  // namespace sieve
