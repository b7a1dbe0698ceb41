// rq.cu -- RaBitQ-style codes of an index on the device (the paper's local
// search over IVF_RQ7 codes: RaBitQ with 7 bits, Sec. 3.1 and Sec. 6.1).
//
// For a row x of partition p, with r = x - c_p, a d x d orthogonal rotation P:
//   o = r / |r|,  o' = P^T o,  D = 2 max_i |o'_i| / (2^bits - 1),
//   mid = (2^bits - 1) / 2,  u_i = rint(o'_i / D + mid) clamped to [0, 2^bits - 1],
//   f = |r| / <u - mid, o'>;
// the estimate of <q, x> is <q, c_p> + f <u - mid, q'> with q' = P^T q.
//
//   k_rq_encode    codes and factors of the rows.  Every sum runs in fp64 in
//                  index order with fused multiply-adds and every division
//                  and square root is correctly rounded, so the codes are a
//                  deterministic function of the rows, the same on any
//                  implementation that keeps that order.
//   k_rq_fill      the code layout the tensor-core scan streams: per block of
//                  128 rows and K-block of 64 elements, 16 KB of fp16 (u - mid)
//                  (half-integers, exact in fp16) in the swizzled byte order of
//                  the shared-memory operand tile; and the factors x 2^-8 in
//                  the same block order, 0 on padding rows.
//   k_rq_rotate    q' = P^T q for a query batch on the tensor cores: the bulk
//                  pipeline with the columns of P as B rows (the three-product
//                  fp16 split of fp32), written out as fp32 rows.
#include "tc_bulk.cuh"

namespace sieve {

constexpr int kRqEncRows = 16;         // rows per pass of an encoder block
constexpr int kRqEncThreads = 256;     // one thread per rotated coordinate (d <= 256)

// the partition of row r: off[p] <= r < off[p + 1] (off nondecreasing)
__device__ __forceinline__ int64_t part_of(const int64_t *off, int64_t nlist, int64_t r) {
    int64_t lo = 0, hi = nlist;   // off[lo] <= r < off[hi]
    while (hi - lo > 1) {
        const int64_t m = (lo + hi) >> 1;
        if (off[m] <= r) lo = m; else hi = m;
    }
    return lo;
}

__global__ void __launch_bounds__(kRqEncThreads) k_rq_encode(
    const float *__restrict__ X, const int64_t *__restrict__ off, int64_t nlist, int64_t n, int d,
    const float *__restrict__ C, const double *__restrict__ P, int bits, uint8_t *__restrict__ codes,
    float *__restrict__ factors) {
    __shared__ double o[kRqEncRows][kRqEncThreads];   // residuals, then the rotated units
    __shared__ uint8_t ucode[kRqEncRows][kRqEncThreads];
    __shared__ double s_norm[kRqEncRows], s_delta[kRqEncRows];
    __shared__ double s_wmax[kRqEncRows][kRqEncThreads / 32];
    __shared__ int64_t s_part[kRqEncRows];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const double top = (double)((1 << bits) - 1), mid = top / 2.0;
    for (int64_t r0 = (int64_t)blockIdx.x * kRqEncRows; r0 < n; r0 += (int64_t)gridDim.x * kRqEncRows) {
        if (tid < kRqEncRows) s_part[tid] = r0 + tid < n ? part_of(off, nlist, r0 + tid) : 0;
        __syncthreads();
        for (int u = tid; u < kRqEncRows * d; u += blockDim.x) {
            const int i = u / d, j = u % d;
            const int64_t row = r0 + i;
            o[i][j] = row < n ? (double)X[row * d + j] - (double)C[s_part[i] * d + j] : 0.0;
        }
        __syncthreads();
        if (tid < kRqEncRows) {   // |r|^2 in index order
            double nn = 0.0;
            for (int j = 0; j < d; ++j) nn = fma(o[tid][j], o[tid][j], nn);
            s_norm[tid] = sqrt(nn);
        }
        __syncthreads();
        for (int u = tid; u < kRqEncRows * d; u += blockDim.x) {
            const int i = u / d, j = u % d;
            if (s_norm[i] != 0.0) o[i][j] = o[i][j] / s_norm[i];
        }
        __syncthreads();
        // o'_t = sum_j P[j][t] o_j, in index order, for every row of the pass
        double acc[kRqEncRows];
#pragma unroll
        for (int i = 0; i < kRqEncRows; ++i) acc[i] = 0.0;
        if (tid < d) {
            for (int j = 0; j < d; ++j) {
                const double pj = P[(int64_t)j * d + tid];
#pragma unroll
                for (int i = 0; i < kRqEncRows; ++i) acc[i] = fma(pj, o[i][j], acc[i]);
            }
        }
        __syncthreads();   // every thread is done reading the units
#pragma unroll
        for (int i = 0; i < kRqEncRows; ++i) {
            if (tid < d) o[i][tid] = acc[i];
            double m = tid < d ? fabs(acc[i]) : 0.0;   // max |o'_t| (exact in any order)
#pragma unroll
            for (int w = 16; w > 0; w >>= 1) m = fmax(m, __shfl_xor_sync(0xffffffffu, m, w));
            if (lane == 0) s_wmax[i][warp] = m;
        }
        __syncthreads();
        if (tid < kRqEncRows) {
            double m = 0.0;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = fmax(m, s_wmax[tid][w]);
            s_delta[tid] = 2.0 * m / top;
        }
        __syncthreads();
        if (tid < d) {
#pragma unroll
            for (int i = 0; i < kRqEncRows; ++i) {
                const int64_t row = r0 + i;
                uint8_t c;
                if (s_norm[i] == 0.0) {
                    c = (uint8_t)rint(mid);
                } else {
                    double v = rint(o[i][tid] / s_delta[i] + mid);
                    v = v < 0.0 ? 0.0 : (v > top ? top : v);
                    c = (uint8_t)v;
                }
                ucode[i][tid] = c;
                if (row < n) codes[row * d + tid] = c;
            }
        }
        __syncthreads();
        if (tid < kRqEncRows && r0 + tid < n) {   // f = |r| / <u - mid, o'>, in index order
            float f = 0.f;
            if (s_norm[tid] != 0.0) {
                double dot = 0.0;
                for (int t = 0; t < d; ++t) dot = fma((double)ucode[tid][t] - mid, o[tid][t], dot);
                f = (float)(s_norm[tid] / dot);
            }
            factors[r0 + tid] = f;
        }
        __syncthreads();
    }
}

// one thread per (block, K-block, row, 16-byte chunk of 8 elements)
__global__ void k_rq_fill(const uint8_t *__restrict__ codes, const float *__restrict__ factors,
                          const int64_t *__restrict__ off, int64_t nparts,
                          const int64_t *__restrict__ blk_off, int d, int nkb, float mid,
                          unsigned char *__restrict__ out, float *__restrict__ fac_out) {
    const int64_t nblocks = blk_off[nparts];
    const int64_t total = nblocks * nkb * kTcRows * 8;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(u & 7);
        const int r = (int)((u >> 3) & (kTcRows - 1));
        const int64_t bk = u >> 10;               // block * nkb + kb
        const int kb = (int)(bk % nkb);
        const int64_t blk = bk / nkb;
        int64_t lo_p = 0, hi_p = nparts;          // partition: blk_off[p] <= blk < blk_off[p + 1]
        while (hi_p - lo_p > 1) {
            const int64_t m = (lo_p + hi_p) >> 1;
            if (blk_off[m] <= blk) lo_p = m; else hi_p = m;
        }
        const int64_t row = off[lo_p] + (blk - blk_off[lo_p]) * kTcRows + r;
        const bool valid = row < off[lo_p + 1];
        uint32_t h[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            float x[2];
#pragma unroll
            for (int b = 0; b < 2; ++b) {
                const int col = kb * 64 + c * 8 + 2 * e + b;
                x[b] = (valid && col < d) ? (float)codes[row * d + col] - mid : 0.f;
            }
            const __half2 hv = __floats2half2_rn(x[0], x[1]);   // exact: half-integers below 128
            h[e] = *reinterpret_cast<const uint32_t *>(&hv);
        }
        unsigned char *dst = out + bk * (int64_t)tcb::kKbBytesHi + (int64_t)r * 128 + ((c ^ (r & 7)) << 4);
        *reinterpret_cast<uint4 *>(dst) = make_uint4(h[0], h[1], h[2], h[3]);
        // the factors scaled by 2^-8 (exact): the scan's accumulator holds
        // <u - mid, q'> x 2^8, so f x 2^-8 turns it into f <u - mid, q'>
        if (kb == 0 && c == 0) fac_out[blk * kTcRows + r] = valid ? factors[row] * (1.f / 256.f) : 0.f;
    }
}

// the tensor-core layout of P^T (row t = column t of P, rounded to fp32): one
// thread per (block, K-block, row, 16-byte chunk), as tc_layout.cu's fill
__global__ void k_rot_fill(const double *__restrict__ P, int d, int nkb, unsigned char *__restrict__ out) {
    const int64_t total = ceil_div(d, kTcRows) * nkb * kTcRows * 8;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total;
         u += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(u & 7);
        const int r = (int)((u >> 3) & (kTcRows - 1));
        const int64_t bk = u >> 10;
        const int kb = (int)(bk % nkb);
        const int t = (int)(bk / nkb) * kTcRows + r;
        float x[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int j = kb * 64 + c * 8 + e;
            x[e] = (t < d && j < d) ? (float)P[(int64_t)j * d + t] : 0.f;
        }
        uint4 h, l;
        tcp::split2(x[0], x[1], h.x, l.x);
        tcp::split2(x[2], x[3], h.y, l.y);
        tcp::split2(x[4], x[5], h.z, l.z);
        tcp::split2(x[6], x[7], h.w, l.w);
        unsigned char *dst = out + bk * kTcBlockBytes + (int64_t)r * 128 + ((c ^ (r & 7)) << 4);
        *reinterpret_cast<uint4 *>(dst) = h;
        *reinterpret_cast<uint4 *>(dst + kTcBlockBytes / 2) = l;
    }
}

// ---------------------------------------------------------------------------
// q' = P^T q on the tensor cores: tiles of 128 queries against the d columns
// of P (B rows in the tensor-core layout of the matrix P^T)
struct RotArgs {
    const float *Q;
    int64_t nq;
    int d;
    const unsigned char *rot;   // tensor-core layout of P^T (row t = column t of P)
    float *Qrot;                // [nq][d] out
    int *status;
    int stages;                 // B stages of the bulk pipeline
};

__device__ int g_rot_status_sink;

struct RotMode {
    using Args = RotArgs;
    static constexpr int kN = 128;
    struct Tile {
        int64_t q0;
        int ni;
        int64_t nb;    // B rows: d
    };
    __device__ static int num_tiles(const Args &a) { return (int)ceil_div(a.nq, tcp::kM); }
    __device__ static int *tile_counter(const Args &) { return nullptr; }
    __device__ static int d(const Args &a) { return a.d; }
    __device__ static int *status(const Args &a) { return a.status ? a.status : &g_rot_status_sink; }
    __device__ static Tile tile(const Args &a, int t) {
        Tile T;
        T.q0 = (int64_t)t * tcp::kM;
        T.ni = (int)(a.nq - T.q0 < tcp::kM ? a.nq - T.q0 : tcp::kM);
        T.nb = a.d;
        return T;
    }
    __device__ static const float *a_row(const Args &a, const Tile &T, int i) {
        return i < T.ni ? a.Q + (T.q0 + i) * a.d : nullptr;
    }
    __device__ static const unsigned char *b_block(const Args &a, const Tile &, int ch) {
        return a.rot + (int64_t)ch * ((a.d + 63) / 64) * kTcBlockBytes;
    }
    struct Epi {
        float *row;
        __device__ void begin(const Args &a, const Tile &T, int slot, unsigned char *) {
            row = slot < T.ni ? a.Qrot + (T.q0 + slot) * a.d : nullptr;
        }
        // v: 32 coordinates of q' x 2^16 (d % 4 == 0, so ncol is a multiple of 4)
        __device__ void chunk(const Args &, const Tile &, int64_t col0, const float (&v)[32], int ncol) {
            if (!row) return;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (4 * j < ncol)
                    *reinterpret_cast<float4 *>(row + col0 + 4 * j) =
                        make_float4(v[4 * j] * tcp::kUnscale, v[4 * j + 1] * tcp::kUnscale,
                                    v[4 * j + 2] * tcp::kUnscale, v[4 * j + 3] * tcp::kUnscale);
        }
        __device__ void prefetch(const Args &, const Tile &, int) {}
        __device__ void start(const Args &, const Tile &, int) {}
        __device__ void end(const Args &, const Tile &) {}
    };
};

__global__ void __launch_bounds__(tcb::kThreads, 1) k_rq_rotate(RotArgs a) {
    extern __shared__ unsigned char smem_raw[];
    tcb::run_bulk<RotMode>(a, smem_raw, a.stages);
}

int rq_nkb(int d) { return (int)ceil_div(d, 64); }

cudaError_t launch_rq_rotation_layout(const double *P, int d, unsigned char *out, cudaStream_t st) {
    k_rot_fill<<<num_sms(), 256, 0, st>>>(P, d, rq_nkb(d), out);
    return cudaGetLastError();
}

size_t rq_rows_bytes(int64_t nblocks, int d) { return (size_t)nblocks * rq_nkb(d) * tcb::kKbBytesHi; }

cudaError_t launch_rq_encode(const float *X, const int64_t *off, int64_t nlist, int64_t n, int d,
                             const float *C, const double *P, int bits, uint8_t *codes, float *factors,
                             cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    const int64_t want = ceil_div(n, kRqEncRows), cap = 8 * (int64_t)num_sms();
    k_rq_encode<<<(unsigned)(want < cap ? want : cap), kRqEncThreads, 0, st>>>(X, off, nlist, n, d, C, P,
                                                                            bits, codes, factors);
    return cudaGetLastError();
}

cudaError_t launch_rq_layout(const uint8_t *codes, const float *factors, const int64_t *off,
                             int64_t nparts, int d, int bits, int64_t *blk_off, unsigned char *out,
                             float *fac_out, cudaStream_t st) {
    launch_tc_block_scan(off, nparts, blk_off, st);
    const float mid = (float)((1 << bits) - 1) * 0.5f;
    k_rq_fill<<<16 * num_sms(), 256, 0, st>>>(codes, factors, off, nparts, blk_off, d, rq_nkb(d), mid,
                                              out, fac_out);
    return cudaGetLastError();
}

static int rq_rotate_stages(int d) { return tcb::stages_for((int)ceil_div(d, 64), 0, 232448 - 128); }

size_t rq_rotate_smem(int d) { return tcb::smem_bytes(rq_rotate_stages(d), 0); }

cudaError_t prepare_rq_rotate(int d) {
    return cudaFuncSetAttribute(k_rq_rotate, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)rq_rotate_smem(d));
}

cudaError_t launch_rq_rotate(const float *Q, int64_t nq, int d, const unsigned char *rot, float *Qrot,
                             int *status, cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    RotArgs a{Q, nq, d, rot, Qrot, status, rq_rotate_stages(d)};
    const int64_t tiles = ceil_div(nq, tcp::kM);
    const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
    k_rq_rotate<<<grid, tcb::kThreads, rq_rotate_smem(d), st>>>(a);
    return cudaGetLastError();
}

}  // namespace sieve
