// common.cuh -- device helpers shared by the libsieve kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "sieve.h"

namespace sieve {

constexpr int kMaxK = 64;        // results per query
constexpr int kMaxD = 1024;      // vector dimension
constexpr int kRqMaxD = 256;     // quantized search: the query tile's split lives in tensor memory
constexpr int kMaxNprobe = 512;  // partitions per query

// SIMT contraction tile: QT queries x RT rows per thread block of 128 threads;
// each thread owns a 4 x 4 block of scores (queries tq + 8a, rows tr + 16b).
constexpr int QT = 32;
constexpr int RT = 64;
constexpr int DK = 64;           // d columns per pipeline stage
constexpr int LDX = DK + 4;      // padded row stride of a staged row chunk
constexpr int kThreads = 128;

// Device control block of one search call (in the caller's workspace).
struct Ctl {
    int n_items;       // items claimed this round (can exceed the cap; clamp on read)
    int n_active;      // active-list entries this round
    int n_tiles;       // scan tiles this round
    int tile_next;     // scan work counter
    int n_deferred;    // queries cut short by the per-round cap
    int n_continue;    // queries with committed ranks left after the merge
    int round;         // rounds finished
    int status;        // 0 or a SIEVE_E* code
    int more;          // 1 while another round is needed
    int n_tc_tiles;    // tensor-core scan tiles this round
    int tc_tile_next;  // tensor-core scan work counter
    int pad[5];
    unsigned long long tot_items, tot_groups, tot_tiles, tot_rows, tot_pairs;
    unsigned long long tot_rows_tc, tot_pairs_tc;   // the tensor-core share of the two above
};

__host__ __device__ inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
__host__ __device__ inline int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

// (sa, ia) ranks before (sb, ib) in the result order: score desc, id asc.
template <typename I>
__device__ __forceinline__ bool ranks_before(float sa, I ia, float sb, I ib) {
    return sa > sb || (sa == sb && ia < ib);
}

__device__ __forceinline__ unsigned lane_id() { return threadIdx.x & 31u; }

// v[j] for a j known only at run time, by a tree of selects (no local memory)
__device__ __forceinline__ float pick32(const float (&v)[32], int j) {
    float t16[16], t8[8], t4[4];
#pragma unroll
    for (int i = 0; i < 16; ++i) t16[i] = (j & 16) ? v[i + 16] : v[i];
#pragma unroll
    for (int i = 0; i < 8; ++i) t8[i] = (j & 8) ? t16[i + 8] : t16[i];
#pragma unroll
    for (int i = 0; i < 4; ++i) t4[i] = (j & 4) ? t8[i + 4] : t8[i];
    const float t0 = (j & 2) ? t4[2] : t4[0], t1 = (j & 2) ? t4[3] : t4[1];
    return (j & 1) ? t1 : t0;
}

// max(a, b, c) in one instruction (the three-input form of max.f32 on
// sm_100-family GPUs); a NaN input is ignored as by fmaxf
__device__ __forceinline__ float fmax3f(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// the largest of 32 values: a tree of three-input maxima (16 instructions)
__device__ __forceinline__ float max_of_32(const float (&v)[32]) {
    float t[11];
#pragma unroll
    for (int i = 0; i < 10; ++i) t[i] = fmax3f(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
    t[10] = fmaxf(v[30], v[31]);
    const float u0 = fmax3f(t[0], t[1], t[2]), u1 = fmax3f(t[3], t[4], t[5]),
                u2 = fmax3f(t[6], t[7], t[8]), u3 = fmaxf(t[9], t[10]);
    return fmaxf(fmax3f(u0, u1, u2), u3);
}

// 16-byte global->shared async copy; src_bytes = 0 zero-fills the destination.
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src, int src_bytes) {
    unsigned dst = static_cast<unsigned>(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(gmem_src),
                 "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// acc[a][b] += sum_t Qs[(tq + 8a) * ldq + c0 + t] * Xs[(tr + 16b) * LDX + t], t = 0 .. DK-1,
// accumulated in increasing t with one fused multiply-add per term.
__device__ __forceinline__ void contract_chunk(float (&acc)[4][4], const float *__restrict__ Qs,
                                               int ldq, int c0, const float *__restrict__ Xs,
                                               int tq, int tr) {
#pragma unroll 4
    for (int t = 0; t < DK; t += 4) {
        float4 qv[4], xv[4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
            qv[a] = *reinterpret_cast<const float4 *>(Qs + (tq + 8 * a) * ldq + c0 + t);
#pragma unroll
        for (int b = 0; b < 4; ++b)
            xv[b] = *reinterpret_cast<const float4 *>(Xs + (tr + 16 * b) * LDX + t);
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                float s = acc[a][b];
                s = fmaf(qv[a].x, xv[b].x, s);
                s = fmaf(qv[a].y, xv[b].y, s);
                s = fmaf(qv[a].z, xv[b].z, s);
                s = fmaf(qv[a].w, xv[b].w, s);
                acc[a][b] = s;
            }
    }
}

// Stage rows [r0, r0 + ROWS) x columns [c0, c0 + DK) of a row-major [nrows][d]
// matrix into Xs[ROWS][LDX]; rows >= nrows and columns >= d are zero-filled.
template <int ROWS = RT>
__device__ __forceinline__ void stage_rows(float *Xs, const float *__restrict__ base, int64_t nrows,
                                           int d, int64_t r0, int c0) {
    constexpr int kVec = DK / 4;
    for (int idx = threadIdx.x; idx < ROWS * kVec; idx += kThreads) {
        int r = idx / kVec, v = idx % kVec;
        int col = c0 + 4 * v;
        bool ok = (r0 + r < nrows) && (col < d);
        const float *src = ok ? base + (r0 + r) * (int64_t)d + col : base;
        cp_async16(Xs + r * LDX + 4 * v, src, ok ? 16 : 0);
    }
}

// Insert (s, id) into a sorted list held in shared memory (capacity cap,
// n = *n_ptr entries, order score desc / id asc).  Called by a full warp with
// warp-uniform arguments; entries falling past cap are dropped.
template <typename I>
__device__ __forceinline__ void warp_list_insert(float *ls, I *li, int *n_ptr, int cap, float s,
                                                 I id) {
    const unsigned lane = lane_id();
    const int n = *n_ptr;
    int pos = 0;
    for (int base = 0; base < n; base += 32) {
        int j = base + lane;
        bool b = j < n && ranks_before(ls[j], li[j], s, id);
        pos += __popc(__ballot_sync(0xffffffffu, b));
    }
    if (pos >= cap) return;
    const int last = n < cap ? n : cap - 1;   // entries [pos, last) move up by one
    for (int base = ((last - 1) / 32) * 32; base >= 0 && last > pos; base -= 32) {
        int j = base + lane;
        bool mv = j >= pos && j < last;
        float vs = mv ? ls[j] : 0.f;
        I vi = mv ? li[j] : I(0);
        __syncwarp();
        if (mv) {
            ls[j + 1] = vs;
            li[j + 1] = vi;
        }
        __syncwarp();
        if (base < pos) break;
    }
    if (lane == 0) {
        ls[pos] = s;
        li[pos] = id;
        *n_ptr = n < cap ? n + 1 : cap;
    }
    __syncwarp();
}

}  // namespace sieve
