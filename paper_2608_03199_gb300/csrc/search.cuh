// search.cuh -- arguments and launchers of the search rounds (internal).
#pragma once

#include <algorithm>

#include "common.cuh"

namespace sieve {

// Everything the round kernels read or write.  Device pointers.
struct SearchArgs {
    // index
    const float *X;            // [n][d] partition-contiguous rows
    const int64_t *ids;        // [n]
    const int64_t *off;        // [nlist+1]
    const float *C;            // [nlist][d] centroids (ranking inside the call)
    int64_t n;
    int64_t nlist;
    int d;
    // queries
    const float *Q;            // [nq][d]
    const int64_t *qids;       // [nq] or nullptr
    const int32_t *order;      // [nq][nprobe]
    int64_t nq;
    // parameters
    float tau;
    int k, nprobe, W, lookahead;
    int serial;                // 1: every (query, rank) item is its own tile (serial traversal)
    int wait_limit;            // polls of the tensor-core scan epilogue's accumulator wait (0: default)
    int64_t cap;               // items per round
    int max_rounds;
    // per-query state: stop line S (Sec. 4.3) and enqueue cursor E (first
    // rank not yet issued), 1-based ranks
    int *S, *E;
    // per-round ready queue
    int *item_q, *item_rank, *item_p;   // [cap]
    int *counts, *cursor;               // [nlist]
    int *bucketed;                      // [cap]
    int4 *tiles;                        // SIMT tiles: partition, first bucketed slot, items
    int4 *tc_tiles;                     // tensor-core tiles (up to 128 items each)
    int tc_min;                         // groups chunks of >= tc_min items go to the
                                        // tensor cores; 0 = SIMT only
    int4 *active;                       // [nq]: query, first item, items
    float *rank_scratch;                // candidate lists of the tensor-core ranking
    const unsigned char *tc_rows;       // tensor-core layout of the rows (nullable)
    const int64_t *tc_row_blocks;       // [nlist+1] block offsets of that layout
    const unsigned char *tc_cent;       // tensor-core layout of the centroids (nullable)
    int tc_stages;                      // B stages of the bulk pipeline (0 = not used)
    int tc_screen;                      // 1: the bulk scan screens with one product per
                                        // pair and rescores candidates in FP32; 0: three
                                        // products per pair
    float *qnorm;                       // [nq] Euclidean norms of the queries (screening)
    // per-item local results
    int *res_cnt;                       // [cap]
    float *res_s;                       // [cap][k]
    long long *res_id;                  // [cap][k]
    // outputs (the running top-k lives here during the search)
    long long *out_ids;
    float *out_scores;
    int *out_count, *out_probes;
    Ctl *ctl;
    // optional provenance (window calibration): the 1-based rank each kept
    // result came from [nq][k], and one bit per rank that held a qualifying
    // row [nq][hit_words]
    int *out_rank;
    unsigned *hit_bits;
    int hit_words;
    // quantized local search over RaBitQ-style codes (rq = 1): the estimate
    // of <q, x> for row x of partition p is cscores(q, rank of p) + f_x
    // <u_x - mid, q'>; rq = 0: exact inner products
    int rq;
    const float *Qrot;                  // [nq][d] rotated queries q' = P^T q
    float *cscores;                     // [nq][nprobe] centroid scores of the ranking
    const unsigned char *rq_rows;       // code layout: fp16 (u - mid), 16 KB per block K-block
    const int64_t *rq_row_blocks;       // [nlist+1] block offsets of that layout
    const float *rq_fac;                // [blocks * 128] factors f in block order
    const unsigned char *rq_rot;        // tensor-core layout of P^T (the query rotation)
};

size_t scan_smem_bytes(int d, int k);
int num_sms();
int scan_blocks_for(size_t smem);
cudaError_t prepare_scan_kernel(size_t smem);
cudaError_t launch_init(const SearchArgs &a, cudaStream_t st);
cudaError_t launch_finalize(const SearchArgs &a, cudaStream_t st);
cudaError_t launch_round(const SearchArgs &a, size_t scan_smem, int scan_blocks,
                         cudaGraphConditionalHandle cond, int use_cond, cudaStream_t st,
                         cudaEvent_t *ev = nullptr);
constexpr int kRoundKernels = 7;   // issue, bucket, scatter, scan_tc, scan, merge, round_end

// tensor-core scan (scan_tc.cu)
constexpr int kTcTile = 128;       // items per tensor-core tile
size_t scan_tc_smem_bytes(int k);
bool scan_tc_fits(int k);          // the converter pipeline's shared memory holds k-lists
cudaError_t prepare_scan_tc(int k);
void enqueue_scan_tc(const SearchArgs &a, cudaStream_t st);
// the same fed from the tensor-core layout by bulk copies (d <= 256)
int scan_bulk_stages(int d, int k);              // 0 when it does not apply
cudaError_t prepare_scan_bulk(int d, int k, int stages);
// the screening variant (a.tc_screen = 1): hi halves of B only, one product
int scan_screen_stages(int d, int k);            // 0 when it does not apply
cudaError_t prepare_scan_screen(int d, int k, int stages);
void enqueue_scan_bulk(const SearchArgs &a, cudaStream_t st);   // either variant

// centroid ranking (rank_kernel.cu): prepare_rank once before launches or
// stream capture, then enqueue_rank (a single kernel launch)
cudaError_t prepare_rank(int nprobe);
// qlist/qlist_n (nullable, device): rank only the listed queries of the nq
// (at most nq of them; the grid covers nq)
cudaError_t enqueue_rank(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                         int nprobe, int32_t *order, float *cscores, cudaStream_t st,
                         const int *qlist = nullptr, const int *qlist_n = nullptr);

// centroid ranking on the tensor cores (rank_tc.cu): one contraction pass with
// a streaming threshold per query, candidate lists of at most
// kRankScratchBytes per chunk of queries, then a warp-per-query selection
constexpr int64_t kRankScratchBytes = int64_t(4) << 30;
bool rank_tc_supported(int64_t nlist, int nprobe);
size_t rank_tc_scratch_bytes(int64_t nq, int64_t nlist, int nprobe, int d);
// kernel launches of one ranking (plan_nq as for enqueue_rank_tc; bulk: the
// centroids' tensor-core layout is given and rank_bulk_stages(d) > 0)
int rank_tc_launches(int64_t nq, int64_t nlist, int nprobe, int d, int64_t plan_nq, bool bulk);
cudaError_t prepare_rank_tc(int nprobe, int d);
// mma_ms (nullable): the contraction launches are bracketed by events, the
// call synchronizes st and adds their summed time (ms) to *mma_ms.
// plan_nq: the query count scratch was sized for (rank_tc_scratch_bytes), when
// these nq queries are a part of that batch; 0 = nq
cudaError_t enqueue_rank_tc(const float *Q, int64_t nq, const float *C, int64_t nlist, int d,
                            int nprobe, int32_t *order, float *cscores, float *scratch, int *status,
                            cudaStream_t st, const unsigned char *tc_cent = nullptr,
                            float *mma_ms = nullptr, int64_t plan_nq = 0);
int rank_tc_mma_launches(int64_t nq, int64_t nlist, int nprobe, int d, int64_t plan_nq,
                         bool bulk);   // contraction launches
int rank_screen_stages(int d);                   // 0 when the screening first pass does not apply
// the first pass's one-product score of every (query, centroid) pair into
// out[q * ld + c] (ld a multiple of 32, out 16-byte aligned, d <= 256)
cudaError_t enqueue_screen_scores(const float *Q, int64_t nq, int64_t nlist, int d,
                                  const unsigned char *tc_cent, float *out, int64_t ld,
                                  int *status, cudaStream_t st);
int rank_bulk_stages(int d);                     // 0 when the bulk ranking does not apply

// in-call window calibration (calibrate.cu)
cudaError_t calib_gather(const float *Q, const int64_t *qids, int d, const int64_t *idx, int64_t n,
                         float *Qo, int64_t *qo, cudaStream_t st);
cudaError_t calib_complement(const int64_t *sample, int64_t ns, int64_t nq, int64_t *rest,
                             cudaStream_t st);
cudaError_t calib_check_sample(const int64_t *sample, int64_t ns, int64_t nq, int *bad,
                               cudaStream_t st);
cudaError_t calib_pick(const unsigned *hit_bits, int words, const int *out_rank, const int *count,
                       int64_t ns, int k, int nprobe, double eps, int fallback,
                       unsigned long long *hist, unsigned long long *Z, int *W_out,
                       cudaStream_t st);
cudaError_t calib_scatter(const int64_t *idx, int64_t n, int k, const long long *ids, const float *sc,
                          const int *cnt, const int *pr, long long *out_ids, float *out_sc,
                          int *out_cnt, int *out_pr, cudaStream_t st);

// the global top-k of several shards' results (shard.cu); per-shard arrays
// are [nshards][nq][k] and [nshards][nq]
cudaError_t launch_merge_shards(int nshards, int64_t nq, int k, const long long *ids, const float *sc,
                                const int *cnt, const int *pr, long long *out_ids, float *out_sc,
                                int *out_cnt, int *out_pr, int *shard_probes, cudaStream_t st);

// tensor-core layout of partition rows and centroids (tc_layout.cu)
constexpr int kTcRows = 128;                   // rows per block
constexpr int64_t kTcBlockBytes = 32768;       // one K-block (64 elements) of a block: hi + lo fp16
int tc_nkb(int d);
size_t tc_norms_bytes(int64_t nblocks);        // the per-block row norms after the blocks
cudaError_t launch_tc_layout_rows(const float *X, const int64_t *off, int64_t nparts, int d,
                                  int64_t *blk_off, unsigned char *out, cudaStream_t st);
cudaError_t launch_tc_layout_matrix(const float *X, int64_t nrows, int d, unsigned char *out,
                                    cudaStream_t st);
// block offsets of the partitions: blk_off[p] = sum over p' < p of ceil(rows / 128)
cudaError_t launch_tc_block_scan(const int64_t *off, int64_t nparts, int64_t *blk_off, cudaStream_t st);

// RaBitQ-style codes (rq.cu): codes and factors of partition-contiguous rows,
// the scan's code layout (16 KB per block K-block, factors in block order),
// and the query rotation q' = P^T q on the tensor cores
int rq_nkb(int d);
size_t rq_rows_bytes(int64_t nblocks, int d);
cudaError_t launch_rq_encode(const float *X, const int64_t *off, int64_t nlist, int64_t n, int d,
                             const float *C, const double *P, int bits, uint8_t *codes, float *factors,
                             cudaStream_t st);
cudaError_t launch_rq_layout(const uint8_t *codes, const float *factors, const int64_t *off,
                             int64_t nparts, int d, int bits, int64_t *blk_off, unsigned char *out,
                             float *fac_out, cudaStream_t st);
cudaError_t launch_rq_rotation_layout(const double *P, int d, unsigned char *out, cudaStream_t st);
cudaError_t prepare_rq_rotate(int d);
cudaError_t launch_rq_rotate(const float *Q, int64_t nq, int d, const unsigned char *rot, float *Qrot,
                             int *status, cudaStream_t st);
// the tensor-core scan over codes (scan_tc.cu)
int scan_rq_stages(int d, int k);                // 0 when it does not apply
cudaError_t prepare_scan_rq(int d, int k, int stages);
void enqueue_scan_rq(const SearchArgs &a, cudaStream_t st);

// partition layout (layout_kernels.cu)
size_t layout_workspace_bytes(int64_t n, int64_t nlist);
cudaError_t launch_layout(const float *X, const int32_t *assign, int64_t n, int d, int64_t nlist,
                          float *X_sorted, int64_t *ids_sorted, int64_t *list_offsets, void *ws,
                          int *bad_flag_host, cudaStream_t st);

}  // namespace sieve
