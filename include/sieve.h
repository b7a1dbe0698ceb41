/*
 * sieve.h -- C ABI of libsieve, a single-GPU (sm_103a) implementation of the
 * data-parallel hot path of SieveIVF's threshold-aware IVF search
 * (arXiv 2608.03199).
 *
 * A query batch Q searches an IVF index: each query ranks the centroids
 * (Sec. 2.3, Sec. 4.1), then visits partitions in that order.  A visit is a
 * hit when the partition holds a row x with sim(q, x) >= tau (R(q, tau),
 * Sec. 2.2).  A query stops after W consecutive empty visits or at nprobe
 * (Sec. 4.1); equivalently it searches ranks 1..s, where the stop line s
 * starts at min(W, nprobe) and a hit at rank j raises it to
 * max(s, min(j + W, nprobe)) (Sec. 4.3).  Active queries are regrouped by
 * partition every round (continuous batching, Algorithm 1); with lookahead
 * every committed rank is issued at once (Algorithm 2).  The result is the
 * top-k of the qualifying rows over the searched partitions (MergeTopK).
 *
 * Conventions for every call:
 *   - similarity is the fp32 inner product of unit-norm vectors (cosine);
 *   - "device" pointers are CUDA global memory of the current device;
 *     "host" pointers are ordinary (ideally page-locked) host memory;
 *   - the library allocates no device memory: scratch comes from the
 *     caller's workspace (ws, ws_bytes), sized by the *_workspace_size calls,
 *     256-byte aligned; the caller owns every buffer and must keep it alive
 *     until the stream has passed the call;
 *   - calls are asynchronous on `stream` (0 = the legacy default stream)
 *     unless stated otherwise; they never abort and never print; a failure
 *     returns a negative sieve_status and, for SIEVE_ECUDA, records the CUDA
 *     error code (sieve_last_cuda_error, per host thread);
 *   - calls on different streams may run concurrently when they use
 *     different workspaces; one workspace must not be shared by calls that
 *     may overlap.
 */
#ifndef SIEVE_H
#define SIEVE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t sieve_status;
#define SIEVE_OK 0
#define SIEVE_EINVAL (-1)       /* bad shape, parameter or null required pointer */
#define SIEVE_ECUDA (-2)        /* a CUDA runtime call failed */
#define SIEVE_EWORKSPACE (-3)   /* ws_bytes below the size the call needs, or ws misaligned */
#define SIEVE_ELIMIT (-4)       /* the device round loop hit its round limit (see sieve_stats) */
#define SIEVE_EUNSUPPORTED (-5) /* the current device is not sm_103 */
#define SIEVE_ESCRATCH (-6)     /* sieve_search_noalloc: the call needs more scratch than
                                   SIEVE_NOALLOC_SCRATCH_BYTES */
#define SIEVE_ETIMEOUT (-7)     /* a bounded device-side wait gave up (reported in sieve_stats) */

/* The IVF index, resident on the device (Sec. 2.3).  Borrowed, read-only.
 *   vectors      device [n][d] fp32, unit-norm, partition-contiguous: the rows
 *                of partition p are list_offsets[p] .. list_offsets[p+1]-1
 *   ids          device [n] int64, the external id of each stored row
 *   list_offsets device [nlist+1] int64, nondecreasing, [0] = 0, [nlist] = n
 *   centroids    device [nlist][d] fp32 (unit-norm for cosine ranking)
 *   tc_rows, tc_row_blocks, tc_centroids  (all nullable) the tensor-core
 *                layout of the rows and of the centroids, made by
 *                sieve_build_tc_layout from this view; when present (and
 *                d <= 256) the tensor-core scan and ranking stream them with
 *                bulk copies instead of splitting fp32 rows on every pass.
 *                They must describe the same vectors and centroids.
 * d must be a multiple of 4 and at most 1024; every base pointer 16-byte
 * aligned.  Every row must sit in the partition of its nearest centroid
 * (exact assignment, the precondition of Sec. 4.4); the library does not
 * check this. */
typedef struct {
    int64_t n;
    int64_t nlist;
    int32_t d;
    int32_t reserved0;
    const float *vectors;
    const int64_t *ids;
    const int64_t *list_offsets;
    const float *centroids;
    const void *tc_rows;
    const int64_t *tc_row_blocks;
    const void *tc_centroids;
} sieve_index_view;

/* Search parameters (Sec. 4, Sec. 6.1).
 *   tau        similarity threshold; a row qualifies iff sim >= tau; not NaN
 *   k          results per query, 1..64
 *   nprobe     maximum partitions per query, 1..min(nlist, 512)
 *   W          consecutive-empty window, >= 1; W >= nprobe is fixed probing
 *   lookahead  0 = continuous batching (one rank per query per round,
 *              Algorithm 1), 1 = issue every committed rank (Algorithm 2)
 *   serial     0 = regroup the ready items by partition every round, up to
 *              128 items per tile (continuous batching, Sec. 4.2); 1 = the
 *              serial traversal of the execution ablation (Sec. 6.3): every
 *              (query, rank) item is its own partition call, one query
 *              against the partition's rows, with the same stopping rule and
 *              the same results; a baseline for measurement
 *   wait_limit iteration limit of one device wait: the tensor-core scan
 *              epilogue's wait for an accumulator (a wait with no
 *              asynchronous work of its own outstanding); 0 = the default,
 *              2^24 polls.  A testing aid for the bounded waits: a wait that
 *              gives up records SIEVE_ETIMEOUT in the call's status word,
 *              the kernel lets every copy and MMA it issued land (those
 *              waits keep their full limit), frees its tensor memory and
 *              returns; the search stops and reports SIEVE_ETIMEOUT.
 *   max_items_per_round  cap on (query, rank) items issued in one round;
 *              0 = automatic.  Only splits work into more rounds: the result
 *              does not depend on it (Sec. 4.2).
 *   loop       0 = device-resident round loop (a CUDA graph whose WHILE node
 *              runs rounds until no item is left; no host sync per round),
 *              1 = host-driven rounds (one stream sync per round; a debugging
 *              aid that must give identical results)
 *   profile    1 = also time every kernel launch with CUDA events recorded on
 *              `stream` around it (implies host-driven rounds and needs a
 *              stats pointer); 0 = no timing
 *   scan_path  which units compute similarities; all paths give the same
 *              decisions up to fp32 rounding (see the parity notes):
 *              0 = automatic (ranking and every partition group on the
 *              tensor cores when the epilogue's k-lists fit: any k with
 *              the tensor-core layout and d <= 256, k <= 22 otherwise; FP32
 *              FMA beyond; with the tensor-core layout the screen below
 *              when tau >= 0.85 and min(W, nprobe) >= 16 or d >= 192,
 *              three products per pair otherwise),
 *              1 = FP32 FMA only, 2 = tensor cores, three products per pair
 *              (SIEVE_EINVAL where they do not fit), 3 = as 2, but with the
 *              tensor-core layout every pair is screened.
 *              The screen: one fp16 product of the hi halves per (query, row) pair, whose
 *              error is bounded by (2^-10 + 2^-12 + d 2^-22) |q| |x| +
 *              2^-26 sqrt(d) (|q| + |x|) (|x| the largest row norm of the
 *              row's 128-row block); only rows whose screened score reaches
 *              the threshold minus that bound are scored again, in fp32 FMA,
 *              and that score decides and is returned.
 */
typedef struct {
    float tau;
    int32_t k;
    int32_t nprobe;
    int32_t W;
    int32_t lookahead;
    int32_t loop;
    int32_t profile;
    int32_t scan_path;
    int32_t serial;
    int32_t wait_limit;
    int64_t max_items_per_round;
} sieve_params;

/* Kernels of one search call, indexing sieve_stats.kernel_ms / kernel_launches:
 * centroid ranking, state initialisation, the issuer, the ready-queue
 * bucketing, the scatter into partition groups, the grouped scan with its
 * fused epilogue on FP32 FMA, the per-query merge, the end-of-round step,
 * finalisation, the grouped scan on the tensor cores, the query rotation
 * of the quantized search (sieve_rq_search), and the score contraction of
 * the tensor-core ranking alone (its launches are also counted, and its time
 * included, under SIEVE_K_RANK). */
enum {
    SIEVE_K_RANK = 0,
    SIEVE_K_INIT,
    SIEVE_K_ISSUE,
    SIEVE_K_BUCKET,
    SIEVE_K_SCATTER,
    SIEVE_K_SCAN,
    SIEVE_K_MERGE,
    SIEVE_K_ROUND_END,
    SIEVE_K_FINALIZE,
    SIEVE_K_SCAN_TC,
    SIEVE_K_RQ_ROTATE,
    SIEVE_K_RANK_MMA,
    SIEVE_NKERNELS
};

/* Counters of one search call (filled only when a stats pointer is given;
 * that makes the call synchronize `stream`).
 *   rounds       rounds executed
 *   items        (query, rank) items searched = sum of probes over queries
 *   groups       sum over rounds of partitions with at least one item
 *                (partition groups, Sec. 4.2); items / groups = mean group
 *   tiles        work tiles of the grouped scan
 *   rows_read    partition rows streamed by the scan (one read per tile)
 *   pairs        query-row similarities computed
 *   rows_read_tc, pairs_tc  the part of rows_read / pairs done on the tensor cores
 *   status       device status word (0, or a SIEVE_E* code) */
typedef struct {
    int64_t rounds;
    int64_t items;
    int64_t groups;
    int64_t tiles;
    int64_t rows_read;
    int64_t pairs;
    int64_t rows_read_tc;
    int64_t pairs_tc;
    int32_t status;
    int32_t reserved0;
    float kernel_ms[SIEVE_NKERNELS];          /* profile = 1: summed launch durations */
    int32_t kernel_launches[SIEVE_NKERNELS];  /* launches per kernel in the call */
} sieve_stats;

/* Partition-contiguous layout of an index (the storage of Sec. 2.3):
 * a stable counting sort of the rows of X by their partition.
 *   X          device [n][d] fp32, rows in any order
 *   assign     device [n] int32, partition of each row, 0 <= assign < nlist
 *   X_sorted   device [n][d] fp32 out; ids_sorted device [n] int64 out (the
 *              row index in X of each sorted row, so the ids are 0..n-1);
 *   list_offsets device [nlist+1] int64 out
 * Rows of one partition keep their order in X.  An out-of-range assign
 * value makes the call return SIEVE_EINVAL after the kernels ran (the call
 * synchronizes `stream`).  Workspace: sieve_layout_workspace_size. */
sieve_status sieve_layout_workspace_size(int64_t n, int64_t nlist, size_t *bytes);
sieve_status sieve_build_layout(const float *X, const int32_t *assign, int64_t n, int32_t d,
                                int64_t nlist, float *X_sorted, int64_t *ids_sorted,
                                int64_t *list_offsets, void *ws, size_t ws_bytes,
                                void *stream);

/* Tensor-core layout of an index: the rows of each partition and the
 * centroids, pre-split for the fp16 contraction (hi = fp16(256 x),
 * lo = fp16(256 x - hi)) and stored in blocks of 128 rows in the byte order
 * of the shared-memory operand tiles (4 bytes per element, each partition
 * padded to a multiple of 128 rows), followed by one fp32 per block of rows:
 * the largest Euclidean norm of its rows (the screening scan's error bound
 * uses it).  Derived data: it changes no result.
 *   sieve_tc_layout_size   bytes of tc_rows and of tc_centroids for this view
 *                          (reads list_offsets from the device: synchronous)
 *   sieve_build_tc_layout  fills tc_rows (device, rows_bytes), tc_row_blocks
 *                          (device [nlist+1] int64, block offsets of the
 *                          partitions) and tc_centroids (device, cent_bytes)
 *                          from ix->vectors, ix->list_offsets, ix->centroids
 * Every output 256-byte aligned; asynchronous on `stream`. */
sieve_status sieve_tc_layout_size(const sieve_index_view *ix, size_t *rows_bytes,
                                  size_t *cent_bytes);
sieve_status sieve_build_tc_layout(const sieve_index_view *ix, void *tc_rows,
                                   int64_t *tc_row_blocks, void *tc_centroids, void *stream);

/* Centroid ranking (Sec. 2.3, Sec. 4.1): for every query, the nprobe
 * centroids with the largest inner product, best first; equal scores rank
 * the lower centroid id first.  Scores come from the tensor cores with the
 * three-product fp16 split (each fp32 value = hi + lo fp16, scaled by 256),
 * accurate to a few 1e-7 on unit vectors.  One contraction pass: the
 * epilogue keeps, per query, a running threshold (a histogram of the scores
 * it has kept) and appends only scores that reach it to a candidate list in
 * the workspace; a warp per query then takes the exact nprobe best of its
 * list.  A list that overflows (many equal scores) sends its query to an
 * exact FP32 ranking.
 *   Q        device [nq][d] fp32
 *   order    device [nq][nprobe] int32 out, 0-based centroid ids
 *   cscores  device [nq][nprobe] fp32 out (nullable): the matching scores
 *   ws       workspace of sieve_rank_workspace_size bytes; SIEVE_EWORKSPACE
 *            if smaller */
sieve_status sieve_rank_workspace_size(const sieve_index_view *ix, int64_t nq, int32_t nprobe,
                                       size_t *bytes);
sieve_status sieve_rank_partitions(const sieve_index_view *ix, const float *Q, int64_t nq,
                                   int32_t nprobe, int32_t *order, float *cscores, void *ws,
                                   size_t ws_bytes, void *stream);

/* The ranking's first-pass score of every (query, centroid) pair: one fp16
 * product of the hi halves of the scaled split (hi = fp16(256 x)), summed in
 * fp32 on the tensor cores -- the screen that bounds the exact scores before
 * the exact pass (the paper has no counterpart: its ranking is exact; this
 * is a diagnostic of this library's arithmetic, used to measure how much of
 * the proven error bound the hardware uses).
 *   ix   needs centroids, tc_centroids and d <= 256
 *   Q    device [nq][d] fp32, 16-byte aligned
 *   out  device [nq][ld] fp32, 16-byte aligned, ld >= nlist and a multiple
 *        of 32; out[q][c] for c < nlist (the rest of a row is not written)
 * Enqueued on `stream`; no workspace, nothing allocated.  SIEVE_EINVAL for a
 * missing layout, d > 256 or a bad ld. */
sieve_status sieve_screen_scores(const sieve_index_view *ix, const float *Q, int64_t nq,
                                 float *out, int64_t ld, void *stream);

/* Workspace bytes sieve_search needs for nq queries with these parameters.
 * host_io = 1 sizes it for sieve_search_host (adds device staging for the
 * queries and results). */
sieve_status sieve_search_workspace_size(const sieve_index_view *ix, int64_t nq,
                                         const sieve_params *p, int32_t host_io,
                                         size_t *bytes);

/* Threshold-aware IVF search (Sec. 4, Algorithms 1 and 2), all on the device.
 *   Q          device [nq][d] fp32 queries (unit-norm)
 *   query_ids  device [nq] int64 (nullable): a row whose id equals its
 *              query's id is neither a candidate nor a hit (self-join
 *              deduplication with queries drawn from the indexed rows)
 *   order      device [nq][nprobe] int32 (nullable): precomputed centroid
 *              ranks; NULL ranks inside the call (sieve_rank_partitions)
 *   out_ids    device [nq][k] int64: result ids by (score desc, id asc),
 *              -1 past out_count
 *   out_scores device [nq][k] fp32: their similarities, -inf past out_count
 *   out_count  device [nq] int32: results per query (<= k)
 *   out_probes device [nq] int32: partitions searched (the final stop line)
 *   stats      host (nullable): counters; non-NULL synchronizes `stream`
 * nq = 0 is valid and does nothing.  A list_offsets table that is not a
 * partition of [0, n), or an order entry outside [0, nlist), is detected on
 * the device: nothing past it is searched and the outputs are undefined.
 * Such a device-side error (SIEVE_EINVAL, or SIEVE_ETIMEOUT / SIEVE_ELIMIT)
 * lands in the status word of the workspace's control block.  The call
 * returns it when it synchronizes anyway: with stats, or with host-driven
 * rounds (p->loop = 1).  Otherwise the call returns as soon as the work is
 * enqueued, and sieve_search_status reads the word afterwards. */
sieve_status sieve_search(const sieve_index_view *ix, const float *Q, int64_t nq,
                          const int64_t *query_ids, const int32_t *order,
                          const sieve_params *p, int64_t *out_ids, float *out_scores,
                          int32_t *out_count, int32_t *out_probes, sieve_stats *stats,
                          void *ws, size_t ws_bytes, void *stream);

/* The device status word of the last search enqueued with workspace ws
 * (sieve_search, or sieve_rq_search, whose workspaces start with the same
 * control block): 0, or the SIEVE_E* code the device recorded.  Copies the
 * word to *status (host) on `stream` and synchronizes `stream`, so call it
 * on the search's stream.  SIEVE_EINVAL for a null or misaligned ws. */
sieve_status sieve_search_status(const void *ws, size_t ws_bytes, int32_t *status, void *stream);

/* sieve_search with the queries and results in HOST memory: copies Q (and
 * query_ids) to device staging inside the workspace, searches, copies the
 * results back and synchronizes `stream` before returning.  Pointers as in
 * sieve_search but host-side; workspace from
 * sieve_search_workspace_size(..., host_io = 1, ...).  The queries go up in
 * up to four chunks on a copy stream that the library creates once per device
 * and host thread (with its events), and each chunk's centroid ranking runs on
 * `stream` as soon as the chunk has landed, so the upload overlaps the
 * ranking (with profile = 1 the upload is one copy and the ranking runs
 * inside the search).  Q_host should be page-locked for the copies to be
 * asynchronous.
 * As the call synchronizes, it returns a device-side error (see
 * sieve_search) with or without stats. */
sieve_status sieve_search_host(const sieve_index_view *ix, const float *Q_host, int64_t nq,
                               const int64_t *query_ids_host, const sieve_params *p,
                               int64_t *out_ids_host, float *out_scores_host,
                               int32_t *out_count_host, int32_t *out_probes_host,
                               sieve_stats *stats, void *ws, size_t ws_bytes, void *stream);

/* sieve_search for callers that cannot allocate device memory at all: a host
 * process without a device allocator, a plug-in whose host application owns
 * every allocation, code that runs while the caller's memory pool is being
 * reset.  The paper has no counterpart; this is a deployment convenience.
 *
 * Arguments and results are those of sieve_search, without the workspace.
 * The caller still provides (and owns) every input and output buffer; the
 * call's scratch is a fixed array of SIEVE_NOALLOC_SCRATCH_BYTES inside the
 * library image, so every GPU that loads the library holds that memory until
 * the process exits.  The call allocates nothing: no cudaMalloc, no CUDA
 * graph (rounds are host-driven, one stream sync per round, whatever
 * p->loop says), no events (p->profile must be 0).
 *   - A call whose scratch need (sieve_search_workspace_size with
 *     host_io = 0) exceeds SIEVE_NOALLOC_SCRATCH_BYTES returns
 *     SIEVE_ESCRATCH and touches nothing.
 *   - Every call looks the array's device address up on the current device
 *     (cudaGetSymbolAddress; the address is not cached, so it stays valid
 *     across a cudaDeviceReset).  Under CUDA's lazy module loading the first
 *     call on a device is the one that loads the library's device code and
 *     so commits the array: that call can fail with an out-of-memory
 *     SIEVE_ECUDA.  A caller that must not fail later makes one small call
 *     at start-up, before any stream capture begins.
 *   - The rounds are host-driven and synchronize `stream`, so a device-side
 *     error (SIEVE_EINVAL for an order entry outside [0, nlist),
 *     SIEVE_ETIMEOUT, SIEVE_ELIMIT) is returned with or without stats.
 *   - Every call on a device uses the same array and leaves its contents
 *     behind; each call initialises what it reads.  Calls that can overlap
 *     on the GPU (other host threads, other streams) race on the array and
 *     must be serialized by the caller.
 * As with sieve_search, the outputs are complete once `stream` has passed
 * the call (the host-driven rounds synchronize `stream` on the way). */
#define SIEVE_NOALLOC_SCRATCH_BYTES ((size_t)64 << 20)
sieve_status sieve_search_noalloc(const sieve_index_view *ix, const float *Q, int64_t nq,
                                  const int64_t *query_ids, const int32_t *order,
                                  const sieve_params *p, int64_t *out_ids, float *out_scores,
                                  int32_t *out_count, int32_t *out_probes, sieve_stats *stats,
                                  void *stream);

/* In-call window calibration (Appendix A, Algorithm 3): the search picks W
 * itself from a sample of the batch.
 *   1. If nq < min_queries or ns == 0, W* = fallback_W and every query runs
 *      with it (the paper's fallback for small calls).
 *   2. The ns sampled queries (sample: device [ns] int64, strictly increasing
 *      row indices of Q; the paper draws them uniformly without replacement)
 *      search all nprobe partitions (fixed probing); their results are final.
 *   3. Each neighbour kept for a sampled query was found at some rank j; the
 *      W-rule reaches rank j iff no run of W empty ranks precedes it, so it
 *      needs W >= 1 + (longest run of empty ranks before j).  H[W] counts the
 *      neighbours by that required window; Z = their total.
 *   4. W* = the smallest W < nprobe with 1 - (H[1] + ... + H[W]) / Z < eps,
 *      else nprobe (full probing); Z == 0: W* = fallback_W.
 *   5. The other nq - ns queries run the search with W = W*.
 * p->W is ignored; p->profile must be 0.  Outputs as sieve_search, for every
 * row of Q (sampled rows report nprobe probes).  W_out (host, required)
 * receives W*; hist_out (host [nprobe + 1], nullable) receives H (H[0] = 0);
 * Z_out (host, nullable) receives Z.  The call synchronizes `stream` once,
 * to read W* back before the second search.  SIEVE_EINVAL if the sample is
 * not strictly increasing rows of Q.  ws: at least
 * sieve_calibrated_search_workspace_size bytes, 256-byte aligned. */
sieve_status sieve_calibrated_search_workspace_size(const sieve_index_view *ix, int64_t nq,
                                                    int64_t ns, const sieve_params *p,
                                                    size_t *bytes);
sieve_status sieve_calibrated_search(const sieve_index_view *ix, const float *Q, int64_t nq,
                                     const int64_t *query_ids, const sieve_params *p,
                                     const int64_t *sample, int64_t ns, double eps,
                                     int64_t min_queries, int32_t fallback_W, int64_t *out_ids,
                                     float *out_scores, int32_t *out_count, int32_t *out_probes,
                                     int32_t *W_out, int64_t *hist_out, int64_t *Z_out, void *ws,
                                     size_t ws_bytes, void *stream);

/* A query batch over nshards independent IVF indexes (the public-100M layout
 * of Sec. 6.1: coarse shards, each with its own IVF index and centroids;
 * the ids of all shards are distinct): every shard runs sieve_search on the
 * whole batch with its own ranking and stopping, with window
 * W_per_shard[s] (host [nshards], nullable: p->W for every shard), and the
 * global top-k by (score desc, id asc) merges the shards' results.
 * out_probes receives the partitions searched over all shards; shard_probes
 * (device [nq][nshards], nullable) each shard's.  Every shard must have the
 * same d and satisfy p (nprobe <= its nlist).  ws: at least
 * sieve_sharded_search_workspace_size bytes, 256-byte aligned. */
sieve_status sieve_sharded_search_workspace_size(const sieve_index_view *shards, int32_t nshards,
                                                 int64_t nq, const sieve_params *p,
                                                 const int32_t *W_per_shard, size_t *bytes);
sieve_status sieve_sharded_search(const sieve_index_view *shards, int32_t nshards, const float *Q,
                                  int64_t nq, const int64_t *query_ids, const sieve_params *p,
                                  const int32_t *W_per_shard, int64_t *out_ids, float *out_scores,
                                  int32_t *out_count, int32_t *out_probes, int32_t *shard_probes,
                                  void *ws, size_t ws_bytes, void *stream);

/* The global top-k of per-shard results (the merge step of
 * sieve_sharded_search, for shards searched by separate calls, e.g. each
 * shard calibrating its own window with sieve_calibrated_search on the same
 * sample, as Appendix A does for the public-100M shards).  Inputs (device):
 * ids/scores [nshards][nq][k] sorted by (score desc, id asc) and padded,
 * count/probes [nshards][nq].  Outputs (device): out_* [nq][k] and [nq]
 * (probes summed over shards); shard_probes [nq][nshards] (nullable).
 * Asynchronous on `stream`. */
sieve_status sieve_merge_shard_results(int32_t nshards, int64_t nq, int32_t k,
                                       const int64_t *ids, const float *scores,
                                       const int32_t *count, const int32_t *probes,
                                       int64_t *out_ids, float *out_scores, int32_t *out_count,
                                       int32_t *out_probes, int32_t *shard_probes, void *stream);

/* ---------------------------------------------------------------------
 * Quantized local search over RaBitQ-style codes (the paper's IVF_RQ7
 * index: RaBitQ configured with 7 bits, Sec. 3.1; the local search of
 * Sec. 6.1).  For a row x of partition p, with r = x - c_p and a d x d
 * orthogonal rotation P (row-major, fp64):
 *   o = r / |r|,  o' = P^T o,  D = 2 max_i |o'_i| / (2^bits - 1),
 *   mid = (2^bits - 1) / 2,
 *   u_i = rint(o'_i / D + mid) clamped to [0, 2^bits - 1]   (the codes)
 *   f   = |r| / <u - mid, o'>                                 (the factor)
 * and the search replaces sim(q, x) by the estimate
 *   <q, c_p> + f <u - mid, q'>,   q' = P^T q,
 * RaBitQ's estimator <o', q'> ~ <o_bar, q'> / <o_bar, o'> (o_bar the
 * normalised code vector) scaled by |r| and shifted by the centroid term.
 * Everything else (ranking, tau, the W-rule, rounds, MergeTopK) is
 * sieve_search's.  These calls need d <= 256 and bits in 1..8.
 * ------------------------------------------------------------------- */

/* Codes and factors of the index's rows (in the view's row order), each
 * row against the centroid of the partition that holds it.
 *   P        device [d][d] fp64, orthogonal (not checked)
 *   codes    device [n][d] uint8 out;  factors device [n] fp32 out
 * Every sum runs in fp64 in index order with fused multiply-adds; divisions
 * and square roots are correctly rounded, so the codes are a deterministic
 * function of the rows.  A row equal to its centroid gets codes rint(mid)
 * and factor 0.  Asynchronous on `stream`. */
sieve_status sieve_rq_encode(const sieve_index_view *ix, const double *P, int32_t bits,
                             uint8_t *codes, float *factors, void *stream);

/* The scan's layout of the codes (derived data, as sieve_build_tc_layout):
 *   rq_rows        per block of 128 rows of a partition and K-block of 64
 *                  elements, 16 KB of fp16 (u - mid) in the byte order of the
 *                  shared-memory operand tile (2 bytes per element)
 *   rq_row_blocks  device [nlist+1] int64, block offsets of the partitions
 *   rq_factors     device [blocks * 128] fp32: the factors x 2^-8 (an exact
 *                  power-of-two scale, the scale of the scan's query split) in
 *                  the same block order, 0 on the padding rows
 *   rq_rotation    the tensor-core layout of P^T (P rounded to fp32), used to
 *                  rotate the queries
 * sieve_rq_layout_size reads list_offsets from the device (synchronous);
 * sieve_build_rq_layout is asynchronous on `stream`.  Outputs 256-byte
 * aligned; codes / factors as made by sieve_rq_encode with the same P. */
sieve_status sieve_rq_layout_size(const sieve_index_view *ix, size_t *rows_bytes,
                                  size_t *factors_bytes, size_t *rotation_bytes);
sieve_status sieve_build_rq_layout(const sieve_index_view *ix, const uint8_t *codes,
                                   const float *factors, int32_t bits, const double *P,
                                   void *rq_rows, int64_t *rq_row_blocks, float *rq_factors,
                                   void *rq_rotation, void *stream);

/* The quantized index beside an index view (borrowed, read-only). */
typedef struct {
    int32_t bits;
    int32_t reserved0;
    const void *rq_rows;
    const int64_t *rq_row_blocks;
    const float *rq_factors;
    const void *rq_rotation;
} sieve_rq_view;

/* sieve_search with the quantized local search: a row qualifies iff its
 * estimate >= tau, and results carry estimates as scores.  The centroid
 * term <q, c_p> is the ranking's score of p: with order == NULL the call
 * ranks (and keeps the scores in the workspace); with a precomputed order,
 * cscores (device [nq][nprobe] fp32, the scores sieve_rank_partitions
 * returns beside it) is required.  Every group runs on the tensor cores
 * (scan_path 1 is SIEVE_EINVAL); ix->tc_rows is not used.  Profiling reports
 * the query rotation under SIEVE_K_RQ_ROTATE.  ws: at least
 * sieve_rq_search_workspace_size bytes, 256-byte aligned. */
sieve_status sieve_rq_search_workspace_size(const sieve_index_view *ix, int64_t nq,
                                            const sieve_params *p, size_t *bytes);
sieve_status sieve_rq_search(const sieve_index_view *ix, const sieve_rq_view *rq, const float *Q,
                             int64_t nq, const int64_t *query_ids, const int32_t *order,
                             const float *cscores, const sieve_params *p, int64_t *out_ids,
                             float *out_scores, int32_t *out_count, int32_t *out_probes,
                             sieve_stats *stats, void *ws, size_t ws_bytes, void *stream);

/* Human-readable name of a status code (static string). */
const char *sieve_status_str(sieve_status s);

/* The CUDA error code behind the calling thread's last SIEVE_ECUDA (0 if none). */
int32_t sieve_last_cuda_error(void);

/* Library version string. */
const char *sieve_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SIEVE_H */
