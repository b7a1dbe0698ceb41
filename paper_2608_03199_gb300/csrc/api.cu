// api.cu -- the C ABI of libsieve (declared in include/sieve.h): argument
// checks, workspace layout, the device-resident round loop as a CUDA graph
// with a WHILE conditional node, and the host-buffer variant.
#include <cstddef>
#include <cstring>
#include <mutex>
#include <vector>

#include "search.cuh"

using namespace sieve;

namespace {

thread_local int32_t g_last_cuda_error = 0;

sieve_status cuda_fail(cudaError_t e) {
    g_last_cuda_error = (int32_t)e;
    return SIEVE_ECUDA;
}

#define SIEVE_CUDA(call)                                  \
    do {                                                  \
        cudaError_t e_ = (call);                          \
        if (e_ != cudaSuccess) return cuda_fail(e_);      \
    } while (0)

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

sieve_status check_device() {
    int dev = 0;
    SIEVE_CUDA(cudaGetDevice(&dev));
    static std::mutex m;
    static std::vector<int> verdict;   // per device: 0 unknown, 1 ok, 2 unsupported
    std::lock_guard<std::mutex> g(m);
    if ((int)verdict.size() <= dev) verdict.resize(dev + 1, 0);
    if (verdict[dev] == 0) {
        int major = 0, minor = 0;
        SIEVE_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
        SIEVE_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
        verdict[dev] = (major == 10 && minor == 3) ? 1 : 2;
    }
    return verdict[dev] == 1 ? SIEVE_OK : SIEVE_EUNSUPPORTED;
}

sieve_status check_index(const sieve_index_view *ix, bool need_centroids) {
    if (!ix) return SIEVE_EINVAL;
    if (ix->n < 0 || ix->nlist < 1 || ix->nlist > INT32_MAX) return SIEVE_EINVAL;
    if (ix->d < 4 || ix->d > kMaxD || ix->d % 4) return SIEVE_EINVAL;
    if (!ix->list_offsets) return SIEVE_EINVAL;
    if (ix->n > 0 && (!ix->vectors || !ix->ids || !aligned16(ix->vectors))) return SIEVE_EINVAL;
    if (need_centroids && (!ix->centroids || !aligned16(ix->centroids))) return SIEVE_EINVAL;
    return SIEVE_OK;
}

sieve_status check_params(const sieve_index_view *ix, const sieve_params *p) {
    if (!p) return SIEVE_EINVAL;
    if (p->tau != p->tau) return SIEVE_EINVAL;   // NaN
    if (p->k < 1 || p->k > kMaxK) return SIEVE_EINVAL;
    if (p->nprobe < 1 || p->nprobe > kMaxNprobe || p->nprobe > ix->nlist) return SIEVE_EINVAL;
    if (p->W < 1) return SIEVE_EINVAL;
    if (p->lookahead != 0 && p->lookahead != 1) return SIEVE_EINVAL;
    if (p->loop != 0 && p->loop != 1) return SIEVE_EINVAL;
    if (p->max_items_per_round < 0) return SIEVE_EINVAL;
    if (p->profile != 0 && p->profile != 1) return SIEVE_EINVAL;
    if (p->scan_path < 0 || p->scan_path > 3) return SIEVE_EINVAL;
    if (p->serial != 0 && p->serial != 1) return SIEVE_EINVAL;
    if (p->wait_limit < 0) return SIEVE_EINVAL;
    return SIEVE_OK;
}

constexpr int kScreenMinWindow = 16;   // automatic scan path: the screen from this window up
constexpr int kScreenMinD = 192;       // ... or at any window from this d up ...
constexpr float kScreenMinTau = 0.85f; // ... and this threshold up (below it nearly every row
                                       // of a probed partition needs its fp32 rescore)
constexpr int64_t kAutoCapMax = int64_t(1) << 24;
constexpr int64_t kCapMax = int64_t(1) << 30;

int64_t items_cap(int64_t nq, const sieve_params *p) {
    const int64_t per = p->lookahead ? std::min<int64_t>(p->W, p->nprobe) : 1;
    const int64_t most = std::max<int64_t>(1, nq * (p->lookahead ? p->nprobe : 1));
    int64_t cap = p->max_items_per_round > 0 ? p->max_items_per_round
                                             : std::min<int64_t>(nq * per, kAutoCapMax);
    cap = std::min(cap, most);
    cap = std::min(cap, kCapMax);
    return std::max<int64_t>(cap, 1);
}

// Byte layout of the search workspace.
struct Layout {
    size_t ctl, order, S, E, counts, cursor, item_q, item_rank, item_p, bucketed, tiles, tc_tiles,
        active, res_cnt, res_s, res_id, rank_scratch, qnorm;
    size_t h_Q, h_qids, h_ids, h_scores, h_count, h_probes, h_status;
    size_t qrot, cscores;   // quantized search: rotated queries, centroid scores
    size_t total;
    int64_t cap, max_tiles;
};

Layout make_layout(const sieve_index_view *ix, int64_t nq, const sieve_params *p, bool host_io,
                   bool rq = false) {
    Layout L{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t at = off;
        off += (size_t)round_up((int64_t)std::max<size_t>(bytes, 1), 256);
        return at;
    };
    const int64_t cap = items_cap(nq, p);
    // SIMT tiles: at most one per QT items plus one per partial chunk; tensor-core
    // tiles: at most one per kTcTile items plus one per partition
    // (serial traversal: one tile per item)
    const int64_t max_tiles = p->serial ? cap + 1
                                        : ceil_div(cap, QT) + ceil_div(cap, kTcTile) + ix->nlist + 1;
    const int64_t max_tc_tiles = p->serial ? cap + 1 : ceil_div(cap, kTcTile) + ix->nlist + 1;
    L.cap = cap;
    L.max_tiles = max_tiles;
    L.ctl = take(sizeof(Ctl));
    L.order = take((size_t)nq * p->nprobe * 4);
    L.S = take((size_t)nq * 4);
    L.E = take((size_t)nq * 4);
    L.counts = take((size_t)ix->nlist * 4);
    L.cursor = take((size_t)ix->nlist * 4);
    L.item_q = take((size_t)cap * 4);
    L.item_rank = take((size_t)cap * 4);
    L.item_p = take((size_t)cap * 4);
    L.bucketed = take((size_t)cap * 4);
    L.tiles = take((size_t)max_tiles * 16);
    L.tc_tiles = take((size_t)max_tc_tiles * 16);
    L.active = take((size_t)nq * 16);
    L.qnorm = take((size_t)nq * 4);
    L.res_cnt = take((size_t)cap * 4);
    L.res_s = take((size_t)cap * p->k * 4);
    L.res_id = take((size_t)cap * p->k * 8);
    L.rank_scratch = (p->scan_path != 1 && rank_tc_supported(ix->nlist, p->nprobe))
                         ? take(rank_tc_scratch_bytes(nq, ix->nlist, p->nprobe, ix->d))
                         : 0;
    if (host_io) {
        L.h_Q = take((size_t)nq * ix->d * 4);
        L.h_qids = take((size_t)nq * 8);
        L.h_ids = take((size_t)nq * p->k * 8);
        L.h_scores = take((size_t)nq * p->k * 4);
        L.h_count = take((size_t)nq * 4);
        L.h_probes = take((size_t)nq * 4);
        L.h_status = take(sizeof(int));
    }
    if (rq) {
        L.qrot = take((size_t)nq * ix->d * 4);
        L.cscores = take((size_t)nq * p->nprobe * 4);
    }
    L.total = off;
    return L;
}

// ---------------------------------------------------------------------------
// CUDA-graph cache: one instantiated graph per distinct argument set (the
// graph bakes every pointer and size in; replaying it for identical arguments
// is exactly what a fresh build would do).
struct GraphKey {
    SearchArgs a;
    int device;
    int with_rank;
    int rank_tc;
    size_t scan_smem;
    int scan_blocks;
    bool operator==(const GraphKey &o) const { return std::memcmp(this, &o, sizeof(*this)) == 0; }
};

struct GraphEntry {
    GraphKey key;
    cudaGraph_t graph;
    cudaGraphExec_t exec;
    uint64_t last_use;
};

std::mutex g_graph_mu;
std::vector<GraphEntry> g_graphs;
uint64_t g_graph_clock = 0;
constexpr size_t kGraphCacheMax = 8;

// the centroid ranking of a search: the tensor-core kernel when it applies,
// reporting a bounded wait that gives up in the search's status word
// (mma_ms, nullable: the contraction's own time is added there; the call syncs)
cudaError_t launch_search_rank(const SearchArgs &a, int rank_tc, cudaStream_t st,
                               float *mma_ms = nullptr) {
    int32_t *order = const_cast<int32_t *>(a.order);
    if (rank_tc)
        return enqueue_rank_tc(a.Q, a.nq, a.C, a.nlist, a.d, a.nprobe, order, a.cscores,
                               a.rank_scratch, &a.ctl->status, st, a.tc_cent, mma_ms);
    return enqueue_rank(a.Q, a.nq, a.C, a.nlist, a.d, a.nprobe, order, a.cscores, st);
}

// quantized search: q' = P^T q for the batch, after init (which clears the
// status word the rotation's bounded waits report to)
cudaError_t launch_search_rotate(const SearchArgs &a, cudaStream_t st) {
    return launch_rq_rotate(a.Q, a.nq, a.d, a.rq_rot, const_cast<float *>(a.Qrot), &a.ctl->status, st);
}

sieve_status build_graph(const GraphKey &key, cudaGraph_t *g_out, cudaGraphExec_t *exec_out) {
    const SearchArgs &a = key.a;
    cudaStream_t cs = nullptr;
    SIEVE_CUDA(cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking));
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaSuccess;
    cudaGraphConditionalHandle cond = 0;
    cudaGraphNodeParams np{};
    cudaGraphNode_t wnode = nullptr;
    do {
        // outer graph: [rank] -> init -> WHILE(rounds) -> finalize
        if ((e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal)) != cudaSuccess) break;
        e = launch_init(a, cs);
        if (e == cudaSuccess && a.rq) e = launch_search_rotate(a, cs);
        if (e == cudaSuccess && key.with_rank) e = launch_search_rank(a, key.rank_tc, cs);
        cudaStreamCaptureStatus cst;
        cudaGraph_t cg = nullptr;
        const cudaGraphNode_t *deps = nullptr;
        size_t ndeps = 0;
        if (e == cudaSuccess)
            e = cudaStreamGetCaptureInfo(cs, &cst, nullptr, &cg, &deps, nullptr, &ndeps);
        if (e == cudaSuccess)
            e = cudaGraphConditionalHandleCreate(&cond, cg, 1, cudaGraphCondAssignDefault);
        if (e == cudaSuccess) {
            np.type = cudaGraphNodeTypeConditional;
            np.conditional.handle = cond;
            np.conditional.type = cudaGraphCondTypeWhile;
            np.conditional.size = 1;
            e = cudaGraphAddNode(&wnode, cg, deps, nullptr, ndeps, &np);
        }
        if (e == cudaSuccess)
            e = cudaStreamUpdateCaptureDependencies(cs, &wnode, nullptr, 1,
                                                    cudaStreamSetCaptureDependencies);
        if (e == cudaSuccess) e = launch_finalize(a, cs);
        cudaError_t e2 = cudaStreamEndCapture(cs, &g);
        if (e == cudaSuccess) e = e2;
        if (e != cudaSuccess) break;
        // loop body: one round
        cudaGraph_t body = np.conditional.phGraph_out[0];
        if ((e = cudaStreamBeginCaptureToGraph(cs, body, nullptr, nullptr, 0,
                                               cudaStreamCaptureModeThreadLocal)) != cudaSuccess)
            break;
        e = launch_round(a, key.scan_smem, key.scan_blocks, cond, 1, cs);
        e2 = cudaStreamEndCapture(cs, &body);
        if (e == cudaSuccess) e = e2;
        if (e != cudaSuccess) break;
        e = cudaGraphInstantiate(exec_out, g, 0);
    } while (0);
    cudaStreamDestroy(cs);
    if (e != cudaSuccess) {
        if (g) cudaGraphDestroy(g);
        return cuda_fail(e);
    }
    *g_out = g;
    return SIEVE_OK;
}

sieve_status run_graph(const GraphKey &key, cudaStream_t st) {
    std::lock_guard<std::mutex> lk(g_graph_mu);
    GraphEntry *hit = nullptr;
    for (auto &ge : g_graphs)
        if (ge.key == key) hit = &ge;
    if (!hit) {
        if (g_graphs.size() >= kGraphCacheMax) {
            size_t victim = 0;
            for (size_t i = 1; i < g_graphs.size(); ++i)
                if (g_graphs[i].last_use < g_graphs[victim].last_use) victim = i;
            cudaGraphExecDestroy(g_graphs[victim].exec);
            cudaGraphDestroy(g_graphs[victim].graph);
            g_graphs.erase(g_graphs.begin() + victim);
        }
        GraphEntry ge{};
        ge.key = key;
        sieve_status rc = build_graph(key, &ge.graph, &ge.exec);
        if (rc != SIEVE_OK) return rc;
        g_graphs.push_back(ge);
        hit = &g_graphs.back();
    }
    hit->last_use = ++g_graph_clock;
    SIEVE_CUDA(cudaGraphLaunch(hit->exec, st));
    return SIEVE_OK;
}

// CUDA events: two around each kernel of a round, two for single launches
struct EventSet {
    cudaEvent_t e[2 * kRoundKernels + 2] = {};
    cudaError_t create() {
        for (auto &x : e) {
            cudaError_t r = cudaEventCreate(&x);
            if (r != cudaSuccess) return r;
        }
        return cudaSuccess;
    }
    ~EventSet() {
        for (auto &x : e)
            if (x) cudaEventDestroy(x);
    }
};

// sieve_search_host's copy stream and events, one set per device and host
// thread (created on first use, kept for the thread's life)
constexpr int kHostChunks = 4;
struct CopyLane {
    bool ok = false;
    cudaError_t err = cudaSuccess;
    int device = -1;
    cudaStream_t stream = nullptr;
    cudaEvent_t start = nullptr, landed[kHostChunks] = {};
};

CopyLane &copy_lane() {
    thread_local std::vector<CopyLane> lanes;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    static CopyLane failed;
    if (e != cudaSuccess) {
        failed.err = e;
        return failed;
    }
    for (auto &l : lanes)
        if (l.device == dev) return l;
    CopyLane l;
    l.device = dev;
    e = cudaStreamCreateWithFlags(&l.stream, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&l.start, cudaEventDisableTiming);
    for (int i = 0; e == cudaSuccess && i < kHostChunks; ++i)
        e = cudaEventCreateWithFlags(&l.landed[i], cudaEventDisableTiming);
    l.ok = e == cudaSuccess;
    l.err = e;
    lanes.push_back(l);
    return lanes.back();
}

// the device-side search on device buffers (shared by sieve_search and
// sieve_search_host); arguments already checked
// optional provenance outputs of a search (window calibration)
struct SearchExtras {
    int32_t *out_rank;    // [nq][k]
    uint32_t *hit_bits;   // [nq][ceil(nprobe / 32)]
};

// quantized local search (sieve_rq_search): the code layout, the rotation's
// layout, and centroid scores given with a precomputed order (else nullptr:
// the ranking writes them into the workspace)
struct RqInputs {
    const sieve_rq_view *v;
    const float *cscores;
};

sieve_status search_device(const sieve_index_view *ix, const float *Q, int64_t nq,
                           const int64_t *qids, const int32_t *order, const sieve_params *p,
                           int64_t *out_ids, float *out_scores, int32_t *out_count,
                           int32_t *out_probes, sieve_stats *stats, unsigned char *ws,
                           const Layout &L, cudaStream_t st, const SearchExtras *ex = nullptr,
                           const RqInputs *rq = nullptr) {
    SearchArgs a;
    std::memset(&a, 0, sizeof(a));   // padding takes part in the graph-cache key
    a.X = ix->vectors;
    a.ids = ix->ids;
    a.off = ix->list_offsets;
    a.C = ix->centroids;
    a.n = ix->n;
    a.nlist = ix->nlist;
    a.d = ix->d;
    a.Q = Q;
    a.qids = qids;
    a.order = order ? order : reinterpret_cast<const int32_t *>(ws + L.order);
    a.nq = nq;
    a.tau = p->tau;
    a.k = p->k;
    a.nprobe = p->nprobe;
    a.W = p->W;
    a.lookahead = p->lookahead;
    a.serial = p->serial;
    a.wait_limit = p->wait_limit;
    a.cap = L.cap;
    a.max_rounds = (int)std::min<int64_t>(INT32_MAX, p->nprobe + ceil_div(nq * p->nprobe, L.cap) + 2);
    a.S = reinterpret_cast<int *>(ws + L.S);
    a.E = reinterpret_cast<int *>(ws + L.E);
    a.item_q = reinterpret_cast<int *>(ws + L.item_q);
    a.item_rank = reinterpret_cast<int *>(ws + L.item_rank);
    a.item_p = reinterpret_cast<int *>(ws + L.item_p);
    a.counts = reinterpret_cast<int *>(ws + L.counts);
    a.cursor = reinterpret_cast<int *>(ws + L.cursor);
    a.bucketed = reinterpret_cast<int *>(ws + L.bucketed);
    a.tiles = reinterpret_cast<int4 *>(ws + L.tiles);
    a.tc_tiles = reinterpret_cast<int4 *>(ws + L.tc_tiles);
    a.active = reinterpret_cast<int4 *>(ws + L.active);
    a.rank_scratch = L.rank_scratch ? reinterpret_cast<float *>(ws + L.rank_scratch) : nullptr;
    a.tc_rows = static_cast<const unsigned char *>(ix->tc_rows);
    a.tc_row_blocks = ix->tc_row_blocks;
    a.tc_cent = static_cast<const unsigned char *>(ix->tc_centroids);
    // the tensor cores take every group when their epilogue's lists fit beside
    // the pipeline's stages: the bulk pipeline (tensor layout, d <= 256) for
    // any k <= 64, the converter pipeline for smaller k
    // with the tensor layout the bulk scan either screens every pair with one
    // product and rescores the candidates, or takes three products per pair.
    // The screen pays per candidate (an fp32 rescore) and saves per pair, so
    // it wins when a round scans many partitions per qualifying row: on the
    // 1M x 256 workload a window of 64 ran 25% faster, one of 8 the same.
    // At small d the three-product scan is bound by its per-chunk overheads
    // rather than the tensor pipe, and screening saves nothing (100M x 96,
    // W = 8: the same time); from d = 192 a window of 8 ran 3% (1M x 256) and
    // 10% (10M x 256) faster screened.  Automatic: the screen from tau 0.85
    // up, at a window of 16 or d >= 192; 2 = three products, 3 = the screen.
    const bool with_layout = a.tc_rows && a.tc_row_blocks;
    const bool screen = with_layout && (p->scan_path == 3 ||
                                        (p->scan_path == 0 && (std::min(p->W, p->nprobe) >= kScreenMinWindow || ix->d >= kScreenMinD) &&
                                         p->tau >= kScreenMinTau));
    const int bulk_stages = !with_layout ? 0
                            : screen    ? scan_screen_stages(ix->d, p->k)
                                        : scan_bulk_stages(ix->d, p->k);
    const bool tc_fits = bulk_stages > 0 || scan_tc_fits(p->k);
    if (p->scan_path >= 2 && !tc_fits) return SIEVE_EINVAL;
    a.tc_min = (p->scan_path == 1 || !tc_fits) ? 0 : 1;
    a.tc_stages = a.tc_min > 0 ? bulk_stages : 0;
    a.tc_screen = (a.tc_stages > 0 && screen) ? 1 : 0;
    a.qnorm = reinterpret_cast<float *>(ws + L.qnorm);
    if (!a.tc_stages) {
        a.tc_rows = nullptr;
        a.tc_row_blocks = nullptr;
    }
    if (rq) {   // every group on the tensor cores, over the codes
        const int rq_stages = scan_rq_stages(ix->d, p->k);
        if (rq_stages == 0 || p->scan_path == 1) return SIEVE_EINVAL;
        a.rq = 1;
        a.tc_min = 1;
        a.tc_stages = rq_stages;
        a.tc_screen = 0;
        a.tc_rows = nullptr;
        a.tc_row_blocks = nullptr;
        a.rq_rows = static_cast<const unsigned char *>(rq->v->rq_rows);
        a.rq_row_blocks = rq->v->rq_row_blocks;
        a.rq_fac = rq->v->rq_factors;
        a.rq_rot = static_cast<const unsigned char *>(rq->v->rq_rotation);
        a.Qrot = reinterpret_cast<const float *>(ws + L.qrot);
        a.cscores = rq->cscores ? const_cast<float *>(rq->cscores) : reinterpret_cast<float *>(ws + L.cscores);
    }
    a.res_cnt = reinterpret_cast<int *>(ws + L.res_cnt);
    a.res_s = reinterpret_cast<float *>(ws + L.res_s);
    a.res_id = reinterpret_cast<long long *>(ws + L.res_id);
    a.out_ids = reinterpret_cast<long long *>(out_ids);
    a.out_scores = out_scores;
    a.out_count = out_count;
    a.out_probes = out_probes;
    a.ctl = reinterpret_cast<Ctl *>(ws + L.ctl);
    if (ex) {
        a.out_rank = ex->out_rank;
        a.hit_bits = ex->hit_bits;
        a.hit_words = (int)ceil_div(p->nprobe, 32);
    }

    const bool with_rank = order == nullptr;
    const int rank_tc = with_rank && a.rank_scratch != nullptr;
    const size_t smem = scan_smem_bytes(ix->d, p->k);
    SIEVE_CUDA(prepare_scan_kernel(smem));
    if (a.rq) {
        SIEVE_CUDA(prepare_scan_rq(ix->d, p->k, a.tc_stages));
        SIEVE_CUDA(prepare_rq_rotate(ix->d));
    } else if (a.tc_min > 0) {
        SIEVE_CUDA(!a.tc_stages   ? prepare_scan_tc(p->k)
                   : a.tc_screen ? prepare_scan_screen(ix->d, p->k, a.tc_stages)
                                 : prepare_scan_bulk(ix->d, p->k, a.tc_stages));
    }
    if (with_rank) SIEVE_CUDA(rank_tc ? prepare_rank_tc(p->nprobe, ix->d) : prepare_rank(p->nprobe));
    const int blocks = scan_blocks_for(smem);

    float ms[SIEVE_NKERNELS] = {0};
    int host_status = 0;   // host-driven rounds: the status word, read with every round's flag
    if (p->loop == 0 && !p->profile) {
        GraphKey key;
        std::memset(&key, 0, sizeof(key));
        key.a = a;
        SIEVE_CUDA(cudaGetDevice(&key.device));
        key.with_rank = with_rank;
        key.rank_tc = rank_tc;
        key.scan_smem = smem;
        key.scan_blocks = blocks;
        sieve_status rc = run_graph(key, st);
        if (rc != SIEVE_OK) return rc;
    } else {
        // host-driven rounds; with profile = 1 every launch is bracketed by
        // CUDA events recorded on the launch stream
        EventSet ev;
        if (p->profile) SIEVE_CUDA(ev.create());
        auto timed = [&](int slot, auto &&launch) -> cudaError_t {
            if (p->profile) cudaEventRecord(ev.e[2 * kRoundKernels], st);
            cudaError_t e = launch();
            if (p->profile) {
                cudaEventRecord(ev.e[2 * kRoundKernels + 1], st);
                cudaEventSynchronize(ev.e[2 * kRoundKernels + 1]);
                float t = 0.f;
                cudaEventElapsedTime(&t, ev.e[2 * kRoundKernels], ev.e[2 * kRoundKernels + 1]);
                ms[slot] += t;
            }
            return e;
        };
        SIEVE_CUDA(timed(SIEVE_K_INIT, [&] { return launch_init(a, st); }));
        if (a.rq) SIEVE_CUDA(timed(SIEVE_K_RQ_ROTATE, [&] { return launch_search_rotate(a, st); }));
        if (with_rank)
            SIEVE_CUDA(timed(SIEVE_K_RANK, [&] {
                return launch_search_rank(a, rank_tc, st, p->profile ? &ms[SIEVE_K_RANK_MMA] : nullptr);
            }));
        for (;;) {
            SIEVE_CUDA(launch_round(a, smem, blocks, 0, 0, st, p->profile ? ev.e : nullptr));
            // the status word and the loop flag are adjacent in the control block
            static_assert(offsetof(Ctl, more) == offsetof(Ctl, status) + sizeof(int), "");
            int word[2] = {0, 0};
            SIEVE_CUDA(cudaMemcpyAsync(word, &a.ctl->status, sizeof(word), cudaMemcpyDeviceToHost, st));
            SIEVE_CUDA(cudaStreamSynchronize(st));
            host_status = word[0];
            const int more = word[1];
            if (p->profile) {
                const int slot[kRoundKernels] = {SIEVE_K_ISSUE, SIEVE_K_BUCKET, SIEVE_K_SCATTER,
                                                 SIEVE_K_SCAN_TC, SIEVE_K_SCAN, SIEVE_K_MERGE,
                                                 SIEVE_K_ROUND_END};
                for (int i = 0; i < kRoundKernels; ++i) {
                    float t = 0.f;
                    SIEVE_CUDA(cudaEventElapsedTime(&t, ev.e[2 * i], ev.e[2 * i + 1]));
                    ms[slot[i]] += t;
                }
            }
            if (!more) break;
        }
        SIEVE_CUDA(timed(SIEVE_K_FINALIZE, [&] { return launch_finalize(a, st); }));
    }
    if (stats) {
        Ctl c;
        SIEVE_CUDA(cudaMemcpyAsync(&c, a.ctl, sizeof(Ctl), cudaMemcpyDeviceToHost, st));
        SIEVE_CUDA(cudaStreamSynchronize(st));
        stats->rounds = c.round;
        stats->items = (int64_t)c.tot_items;
        stats->groups = (int64_t)c.tot_groups;
        stats->tiles = (int64_t)c.tot_tiles;
        stats->rows_read = (int64_t)c.tot_rows;
        stats->pairs = (int64_t)c.tot_pairs;
        stats->rows_read_tc = (int64_t)c.tot_rows_tc;
        stats->pairs_tc = (int64_t)c.tot_pairs_tc;
        stats->status = c.status;
        stats->reserved0 = 0;
        for (int i = 0; i < SIEVE_NKERNELS; ++i) stats->kernel_ms[i] = ms[i];
        const int per_round[] = {SIEVE_K_ISSUE, SIEVE_K_BUCKET, SIEVE_K_SCATTER, SIEVE_K_SCAN,
                                 SIEVE_K_MERGE, SIEVE_K_ROUND_END};
        stats->kernel_launches[SIEVE_K_RANK] =
            !with_rank ? 0
            : rank_tc ? rank_tc_launches(a.nq, a.nlist, a.nprobe, a.d, 0,
                                         a.tc_cent && rank_bulk_stages(a.d) > 0)
                      : 1;
        stats->kernel_launches[SIEVE_K_INIT] = a.tc_screen ? 2 : 1;   // + the query norms
        stats->kernel_launches[SIEVE_K_FINALIZE] = 1;
        for (int slot : per_round) stats->kernel_launches[slot] = c.round;
        stats->kernel_launches[SIEVE_K_SCAN_TC] = a.tc_min > 0 ? c.round : 0;
        stats->kernel_launches[SIEVE_K_RQ_ROTATE] = a.rq ? 1 : 0;
        stats->kernel_launches[SIEVE_K_RANK_MMA] =
            with_rank && rank_tc ? rank_tc_mma_launches(a.nq, a.nlist, a.nprobe, a.d, 0,
                                                         a.tc_cent && rank_bulk_stages(a.d) > 0)
                                  : 0;
        if (a.tc_min == 1) stats->kernel_launches[SIEVE_K_SCAN] = 0;
        if (c.status != 0) return c.status;
    }
    // host-driven rounds synchronize every round anyway: a device error is
    // returned even without stats (in graph mode sieve_search_status reads it)
    return host_status != 0 ? host_status : SIEVE_OK;
}

sieve_status check_search(const sieve_index_view *ix, const float *Q, int64_t nq,
                          const int32_t *order, const sieve_params *p, const void *o1,
                          const void *o2, const void *o3, const void *o4) {
    sieve_status rc = check_index(ix, order == nullptr);
    if (rc != SIEVE_OK) return rc;
    if ((rc = check_params(ix, p)) != SIEVE_OK) return rc;
    if (nq < 0 || nq > INT32_MAX / 2) return SIEVE_EINVAL;
    if (nq > 0 && (!Q || !o1 || !o2 || !o3 || !o4)) return SIEVE_EINVAL;
    return SIEVE_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
extern "C" {

const char *sieve_version(void) { return "libsieve 0.1 (sm_103a)"; }

int32_t sieve_last_cuda_error(void) { return g_last_cuda_error; }

const char *sieve_status_str(sieve_status s) {
    switch (s) {
        case SIEVE_OK: return "ok";
        case SIEVE_EINVAL: return "invalid argument";
        case SIEVE_ECUDA: return "CUDA error";
        case SIEVE_EWORKSPACE: return "workspace too small or misaligned";
        case SIEVE_ELIMIT: return "round limit reached";
        case SIEVE_EUNSUPPORTED: return "unsupported device (needs sm_103)";
        case SIEVE_ESCRATCH: return "call needs more scratch than the fixed no-allocation array";
        case SIEVE_ETIMEOUT: return "a bounded device-side wait gave up";
        default: return "unknown status";
    }
}

sieve_status sieve_layout_workspace_size(int64_t n, int64_t nlist, size_t *bytes) {
    if (!bytes || n < 0 || nlist < 1) return SIEVE_EINVAL;
    *bytes = layout_workspace_bytes(n, nlist);
    return SIEVE_OK;
}

sieve_status sieve_build_layout(const float *X, const int32_t *assign, int64_t n, int32_t d,
                                int64_t nlist, float *X_sorted, int64_t *ids_sorted,
                                int64_t *list_offsets, void *ws, size_t ws_bytes, void *stream) {
    if (n < 0 || nlist < 1 || nlist > INT32_MAX || d < 4 || d % 4 || d > kMaxD) return SIEVE_EINVAL;
    if (!list_offsets) return SIEVE_EINVAL;
    if (n > 0 && (!X || !assign || !X_sorted || !ids_sorted || !aligned16(X) || !aligned16(X_sorted)))
        return SIEVE_EINVAL;
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u)) return SIEVE_EWORKSPACE;
    if (ws_bytes < layout_workspace_bytes(n, nlist)) return SIEVE_EWORKSPACE;
    sieve_status rc = check_device();
    if (rc != SIEVE_OK) return rc;
    int bad = 0;
    SIEVE_CUDA(launch_layout(X, assign, n, d, nlist, X_sorted, ids_sorted, list_offsets, ws, &bad,
                             static_cast<cudaStream_t>(stream)));
    return bad ? SIEVE_EINVAL : SIEVE_OK;
}

sieve_status sieve_tc_layout_size(const sieve_index_view *ix, size_t *rows_bytes,
                                  size_t *cent_bytes) {
    if (!rows_bytes || !cent_bytes) return SIEVE_EINVAL;
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    std::vector<int64_t> off((size_t)ix->nlist + 1);
    SIEVE_CUDA(cudaMemcpy(off.data(), ix->list_offsets, off.size() * sizeof(int64_t),
                          cudaMemcpyDeviceToHost));
    int64_t blocks = 0;
    for (int64_t p = 0; p < ix->nlist; ++p) {
        if (off[p + 1] < off[p]) return SIEVE_EINVAL;
        blocks += ceil_div(off[p + 1] - off[p], kTcRows);
    }
    const int64_t per_block = (int64_t)tc_nkb(ix->d) * kTcBlockBytes;
    *rows_bytes = (size_t)(blocks * per_block) + tc_norms_bytes(blocks);
    *cent_bytes = (size_t)(ceil_div(ix->nlist, kTcRows) * per_block);
    return SIEVE_OK;
}

sieve_status sieve_build_tc_layout(const sieve_index_view *ix, void *tc_rows,
                                   int64_t *tc_row_blocks, void *tc_centroids, void *stream) {
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    if (!tc_rows || !tc_row_blocks || !tc_centroids) return SIEVE_EINVAL;
    if ((reinterpret_cast<uintptr_t>(tc_rows) | reinterpret_cast<uintptr_t>(tc_centroids)) & 255u)
        return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    SIEVE_CUDA(launch_tc_layout_rows(ix->vectors, ix->list_offsets, ix->nlist, ix->d, tc_row_blocks,
                                     static_cast<unsigned char *>(tc_rows), st));
    SIEVE_CUDA(launch_tc_layout_matrix(ix->centroids, ix->nlist, ix->d,
                                       static_cast<unsigned char *>(tc_centroids), st));
    return SIEVE_OK;
}

sieve_status sieve_rank_workspace_size(const sieve_index_view *ix, int64_t nq, int32_t nprobe,
                                       size_t *bytes) {
    if (!bytes) return SIEVE_EINVAL;
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    if (nprobe < 1 || nprobe > kMaxNprobe || nprobe > ix->nlist || nq < 0) return SIEVE_EINVAL;
    *bytes = rank_tc_supported(ix->nlist, nprobe) && nq > 0 ? rank_tc_scratch_bytes(nq, ix->nlist, nprobe, ix->d) : 0;
    return SIEVE_OK;
}

sieve_status sieve_rank_partitions(const sieve_index_view *ix, const float *Q, int64_t nq,
                                   int32_t nprobe, int32_t *order, float *cscores, void *ws,
                                   size_t ws_bytes, void *stream) {
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    if (nprobe < 1 || nprobe > kMaxNprobe || nprobe > ix->nlist) return SIEVE_EINVAL;
    if (nq < 0 || nq > INT32_MAX / 2) return SIEVE_EINVAL;
    if (nq > 0 && (!Q || !order || !aligned16(Q))) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (nq == 0) return SIEVE_OK;
    if (rank_tc_supported(ix->nlist, nprobe)) {
        if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) ||
            ws_bytes < rank_tc_scratch_bytes(nq, ix->nlist, nprobe, ix->d))
            return SIEVE_EWORKSPACE;
        SIEVE_CUDA(prepare_rank_tc(nprobe, ix->d));
        SIEVE_CUDA(enqueue_rank_tc(Q, nq, ix->centroids, ix->nlist, ix->d, nprobe, order, cscores,
                                   static_cast<float *>(ws), nullptr,
                                   static_cast<cudaStream_t>(stream),
                                   static_cast<const unsigned char *>(ix->tc_centroids)));
    } else {
        SIEVE_CUDA(prepare_rank(nprobe));
        SIEVE_CUDA(enqueue_rank(Q, nq, ix->centroids, ix->nlist, ix->d, nprobe, order, cscores,
                                static_cast<cudaStream_t>(stream)));
    }
    return SIEVE_OK;
}

sieve_status sieve_screen_scores(const sieve_index_view *ix, const float *Q, int64_t nq,
                                 float *out, int64_t ld, void *stream) {
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    if (!ix->tc_centroids || ix->d > 256) return SIEVE_EINVAL;
    if (nq < 0 || nq > INT32_MAX / 2) return SIEVE_EINVAL;
    if (ld < ix->nlist || ld % 32 != 0 || ld > INT32_MAX) return SIEVE_EINVAL;
    if (nq > 0 && (!Q || !out || !aligned16(Q) || !aligned16(out))) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (nq == 0) return SIEVE_OK;
    SIEVE_CUDA(enqueue_screen_scores(Q, nq, ix->nlist, ix->d,
                                     static_cast<const unsigned char *>(ix->tc_centroids), out, ld,
                                     nullptr, static_cast<cudaStream_t>(stream)));
    return SIEVE_OK;
}

sieve_status sieve_search_workspace_size(const sieve_index_view *ix, int64_t nq,
                                         const sieve_params *p, int32_t host_io, size_t *bytes) {
    if (!bytes) return SIEVE_EINVAL;
    sieve_status rc = check_index(ix, false);
    if (rc != SIEVE_OK) return rc;
    if ((rc = check_params(ix, p)) != SIEVE_OK) return rc;
    if (nq < 0 || nq > INT32_MAX / 2) return SIEVE_EINVAL;
    *bytes = make_layout(ix, nq, p, host_io != 0).total;
    return SIEVE_OK;
}

sieve_status sieve_search(const sieve_index_view *ix, const float *Q, int64_t nq,
                          const int64_t *query_ids, const int32_t *order, const sieve_params *p,
                          int64_t *out_ids, float *out_scores, int32_t *out_count,
                          int32_t *out_probes, sieve_stats *stats, void *ws, size_t ws_bytes,
                          void *stream) {
    sieve_status rc = check_search(ix, Q, nq, order, p, out_ids, out_scores, out_count, out_probes);
    if (rc != SIEVE_OK) return rc;
    if (nq > 0 && !aligned16(Q)) return SIEVE_EINVAL;
    if (p->profile && !stats) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (stats) std::memset(stats, 0, sizeof(*stats));
    if (nq == 0) return SIEVE_OK;
    const Layout L = make_layout(ix, nq, p, false);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < L.total)
        return SIEVE_EWORKSPACE;
    return search_device(ix, Q, nq, query_ids, order, p, out_ids, out_scores, out_count,
                         out_probes, stats, static_cast<unsigned char *>(ws), L,
                         static_cast<cudaStream_t>(stream));
}

sieve_status sieve_search_status(const void *ws, size_t ws_bytes, int32_t *status, void *stream) {
    if (!ws || !status || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < sizeof(Ctl))
        return SIEVE_EINVAL;
    // the control block opens every search layout (make_layout's first part)
    const Ctl *ctl = static_cast<const Ctl *>(ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int32_t v = 0;
    SIEVE_CUDA(cudaMemcpyAsync(&v, &ctl->status, sizeof(v), cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaStreamSynchronize(st));
    *status = v;
    return SIEVE_OK;
}

// ---------------------------------------------------------------------------
// Quantized local search over RaBitQ-style codes (Sec. 3.1, Sec. 6.1).
static sieve_status check_rq_index(const sieve_index_view *ix, int32_t bits) {
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    if (ix->d > kRqMaxD || bits < 1 || bits > 8) return SIEVE_EINVAL;
    return SIEVE_OK;
}

sieve_status sieve_rq_encode(const sieve_index_view *ix, const double *P, int32_t bits,
                             uint8_t *codes, float *factors, void *stream) {
    sieve_status rc = check_rq_index(ix, bits);
    if (rc != SIEVE_OK) return rc;
    if (!P || (ix->n > 0 && (!codes || !factors))) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    SIEVE_CUDA(launch_rq_encode(ix->vectors, ix->list_offsets, ix->nlist, ix->n, ix->d, ix->centroids, P,
                                bits, codes, factors, static_cast<cudaStream_t>(stream)));
    return SIEVE_OK;
}

sieve_status sieve_rq_layout_size(const sieve_index_view *ix, size_t *rows_bytes,
                                  size_t *factors_bytes, size_t *rotation_bytes) {
    if (!rows_bytes || !factors_bytes || !rotation_bytes) return SIEVE_EINVAL;
    sieve_status rc = check_rq_index(ix, 7);
    if (rc != SIEVE_OK) return rc;
    std::vector<int64_t> off((size_t)ix->nlist + 1);
    SIEVE_CUDA(cudaMemcpy(off.data(), ix->list_offsets, off.size() * sizeof(int64_t),
                          cudaMemcpyDeviceToHost));
    int64_t blocks = 0;
    for (int64_t p = 0; p < ix->nlist; ++p) {
        if (off[p + 1] < off[p]) return SIEVE_EINVAL;
        blocks += ceil_div(off[p + 1] - off[p], kTcRows);
    }
    *rows_bytes = rq_rows_bytes(blocks, ix->d);
    *factors_bytes = (size_t)blocks * kTcRows * sizeof(float);
    *rotation_bytes = (size_t)(ceil_div(ix->d, kTcRows) * (int64_t)tc_nkb(ix->d) * kTcBlockBytes);
    return SIEVE_OK;
}

sieve_status sieve_build_rq_layout(const sieve_index_view *ix, const uint8_t *codes,
                                   const float *factors, int32_t bits, const double *P,
                                   void *rq_rows, int64_t *rq_row_blocks, float *rq_factors,
                                   void *rq_rotation, void *stream) {
    sieve_status rc = check_rq_index(ix, bits);
    if (rc != SIEVE_OK) return rc;
    if (!P || !rq_rows || !rq_row_blocks || !rq_factors || !rq_rotation) return SIEVE_EINVAL;
    if (ix->n > 0 && (!codes || !factors)) return SIEVE_EINVAL;
    if ((reinterpret_cast<uintptr_t>(rq_rows) | reinterpret_cast<uintptr_t>(rq_rotation) |
         reinterpret_cast<uintptr_t>(rq_factors)) & 255u)
        return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    SIEVE_CUDA(launch_rq_layout(codes, factors, ix->list_offsets, ix->nlist, ix->d, bits, rq_row_blocks,
                                static_cast<unsigned char *>(rq_rows), rq_factors, st));
    SIEVE_CUDA(launch_rq_rotation_layout(P, ix->d, static_cast<unsigned char *>(rq_rotation), st));
    return SIEVE_OK;
}

sieve_status sieve_rq_search_workspace_size(const sieve_index_view *ix, int64_t nq,
                                            const sieve_params *p, size_t *bytes) {
    if (!bytes) return SIEVE_EINVAL;
    sieve_status rc = check_rq_index(ix, 7);
    if (rc != SIEVE_OK) return rc;
    if ((rc = check_params(ix, p)) != SIEVE_OK) return rc;
    if (nq < 0 || nq > INT32_MAX / 2) return SIEVE_EINVAL;
    *bytes = make_layout(ix, nq, p, false, true).total;
    return SIEVE_OK;
}

sieve_status sieve_rq_search(const sieve_index_view *ix, const sieve_rq_view *rq, const float *Q,
                             int64_t nq, const int64_t *query_ids, const int32_t *order,
                             const float *cscores, const sieve_params *p, int64_t *out_ids,
                             float *out_scores, int32_t *out_count, int32_t *out_probes,
                             sieve_stats *stats, void *ws, size_t ws_bytes, void *stream) {
    sieve_status rc = check_search(ix, Q, nq, order, p, out_ids, out_scores, out_count, out_probes);
    if (rc != SIEVE_OK) return rc;
    if (!rq || (rc = check_rq_index(ix, rq->bits)) != SIEVE_OK) return SIEVE_EINVAL;
    if (!rq->rq_rows || !rq->rq_row_blocks || !rq->rq_factors || !rq->rq_rotation) return SIEVE_EINVAL;
    if ((reinterpret_cast<uintptr_t>(rq->rq_rows) | reinterpret_cast<uintptr_t>(rq->rq_rotation) |
         reinterpret_cast<uintptr_t>(rq->rq_factors)) & 15u)
        return SIEVE_EINVAL;
    if (order && !cscores) return SIEVE_EINVAL;
    if (p->scan_path == 1 || scan_rq_stages(ix->d, p->k) == 0) return SIEVE_EINVAL;
    if (nq > 0 && !aligned16(Q)) return SIEVE_EINVAL;
    if (p->profile && !stats) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (stats) std::memset(stats, 0, sizeof(*stats));
    if (nq == 0) return SIEVE_OK;
    const Layout L = make_layout(ix, nq, p, false, true);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < L.total)
        return SIEVE_EWORKSPACE;
    const RqInputs in{rq, order ? cscores : nullptr};
    return search_device(ix, Q, nq, query_ids, order, p, out_ids, out_scores, out_count, out_probes,
                         stats, static_cast<unsigned char *>(ws), L, static_cast<cudaStream_t>(stream),
                         nullptr, &in);
}

sieve_status sieve_search_host(const sieve_index_view *ix, const float *Q_host, int64_t nq,
                               const int64_t *query_ids_host, const sieve_params *p,
                               int64_t *out_ids_host, float *out_scores_host,
                               int32_t *out_count_host, int32_t *out_probes_host,
                               sieve_stats *stats, void *ws, size_t ws_bytes, void *stream) {
    sieve_status rc = check_search(ix, Q_host, nq, nullptr, p, out_ids_host, out_scores_host,
                                   out_count_host, out_probes_host);
    if (rc != SIEVE_OK) return rc;
    if (p->profile && !stats) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (stats) std::memset(stats, 0, sizeof(*stats));
    if (nq == 0) return SIEVE_OK;
    const Layout L = make_layout(ix, nq, p, true);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < L.total)
        return SIEVE_EWORKSPACE;
    unsigned char *w = static_cast<unsigned char *>(ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    float *dQ = reinterpret_cast<float *>(w + L.h_Q);
    int64_t *dqids = query_ids_host ? reinterpret_cast<int64_t *>(w + L.h_qids) : nullptr;
    int64_t *dids = reinterpret_cast<int64_t *>(w + L.h_ids);
    float *dsc = reinterpret_cast<float *>(w + L.h_scores);
    int32_t *dcnt = reinterpret_cast<int32_t *>(w + L.h_count);
    int32_t *dpr = reinterpret_cast<int32_t *>(w + L.h_probes);
    int *dstatus = reinterpret_cast<int *>(w + L.h_status);
    int32_t *dorder = reinterpret_cast<int32_t *>(w + L.order);
    // The queries go to the device in chunks on a copy stream, and each
    // chunk's centroid ranking starts as soon as it has landed, so the copy
    // overlaps the ranking; the search then runs with the order it made.
    // Chunks are multiples of 128 x (SMs) queries: whole waves of ranking tiles.
    // (With profile = 1 the ranking stays inside the search, where it is timed.)
    CopyLane &cl = copy_lane();
    if (!cl.ok) return cuda_fail(cl.err);
    const int64_t wave = (int64_t)128 * num_sms();
    const int64_t chunk = round_up(ceil_div(nq, kHostChunks), wave);
    const int nchunks = p->profile ? 0 : (int)std::min<int64_t>(kHostChunks, ceil_div(nq, chunk));
    const bool rank_tc = p->scan_path != 1 && L.rank_scratch != 0;
    SIEVE_CUDA(rank_tc ? prepare_rank_tc(p->nprobe, ix->d) : prepare_rank(p->nprobe));
    SIEVE_CUDA(cudaMemsetAsync(dstatus, 0, sizeof(int), st));
    SIEVE_CUDA(cudaEventRecord(cl.start, st));             // earlier work on the staging
    SIEVE_CUDA(cudaStreamWaitEvent(cl.stream, cl.start, 0));
    // the ids first: a copy queued behind the chunks on the same copy engine
    // would hold the first chunk's ranking back until every chunk had landed
    if (dqids && nchunks)
        SIEVE_CUDA(cudaMemcpyAsync(dqids, query_ids_host, (size_t)nq * 8, cudaMemcpyHostToDevice,
                                   cl.stream));
    for (int c = 0; c < nchunks; ++c) {
        const int64_t q0 = c * chunk, n = std::min<int64_t>(chunk, nq - q0);
        SIEVE_CUDA(cudaMemcpyAsync(dQ + q0 * ix->d, Q_host + q0 * ix->d, (size_t)n * ix->d * 4,
                                   cudaMemcpyHostToDevice, cl.stream));
        SIEVE_CUDA(cudaEventRecord(cl.landed[c], cl.stream));
    }
    if (p->profile)
        SIEVE_CUDA(cudaMemcpyAsync(dQ, Q_host, (size_t)nq * ix->d * 4, cudaMemcpyHostToDevice, st));
    if (dqids && !nchunks)
        SIEVE_CUDA(cudaMemcpyAsync(dqids, query_ids_host, (size_t)nq * 8, cudaMemcpyHostToDevice, st));
    int rank_launches = 0, mma_launches = 0;
    for (int c = 0; c < nchunks; ++c) {
        const int64_t q0 = c * chunk, n = std::min<int64_t>(chunk, nq - q0);
        SIEVE_CUDA(cudaStreamWaitEvent(st, cl.landed[c], 0));
        if (rank_tc)
            SIEVE_CUDA(enqueue_rank_tc(dQ + q0 * ix->d, n, ix->centroids, ix->nlist, ix->d, p->nprobe,
                                       dorder + q0 * p->nprobe, nullptr,
                                       reinterpret_cast<float *>(w + L.rank_scratch), dstatus, st,
                                       static_cast<const unsigned char *>(ix->tc_centroids),
                                       nullptr, nq));
        else
            SIEVE_CUDA(enqueue_rank(dQ + q0 * ix->d, n, ix->centroids, ix->nlist, ix->d, p->nprobe,
                                    dorder + q0 * p->nprobe, nullptr, st));
        const bool bulk = ix->tc_centroids && rank_bulk_stages(ix->d) > 0;
        rank_launches += rank_tc ? rank_tc_launches(n, ix->nlist, p->nprobe, ix->d, nq, bulk) : 1;
        mma_launches += rank_tc ? rank_tc_mma_launches(n, ix->nlist, p->nprobe, ix->d, nq, bulk) : 0;
    }
    rc = search_device(ix, dQ, nq, dqids, nchunks ? dorder : nullptr, p, dids, dsc, dcnt, dpr, stats,
                       w, L, st);
    if (rc != SIEVE_OK) return rc;
    SIEVE_CUDA(cudaMemcpyAsync(out_ids_host, dids, (size_t)nq * p->k * 8, cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaMemcpyAsync(out_scores_host, dsc, (size_t)nq * p->k * 4, cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaMemcpyAsync(out_count_host, dcnt, (size_t)nq * 4, cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaMemcpyAsync(out_probes_host, dpr, (size_t)nq * 4, cudaMemcpyDeviceToHost, st));
    int rank_status = 0, search_status = 0;
    SIEVE_CUDA(cudaMemcpyAsync(&rank_status, dstatus, sizeof(int), cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaMemcpyAsync(&search_status, &reinterpret_cast<const Ctl *>(w + L.ctl)->status,
                               sizeof(int), cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaStreamSynchronize(st));
    if (stats && nchunks > 0) {   // ran here
        stats->kernel_launches[SIEVE_K_RANK] = rank_launches;
        stats->kernel_launches[SIEVE_K_RANK_MMA] = mma_launches;
    }
    return rank_status != 0 ? rank_status : search_status != 0 ? search_status : SIEVE_OK;
}

// ---------------------------------------------------------------------------
// In-call window calibration (Appendix A, Algorithm 3).  Scratch, in order:
// the inner search's workspace (sized for the larger of the two searches, both
// at W = nprobe, the widest window the calibration can pick), then the sample
// and remainder buffers below.
struct CalibLayout {
    Layout inner;
    size_t Qs, qs, s_ids, s_sc, s_cnt, s_pr, s_rank, s_hits, rest, Qr, qr, r_ids, r_sc, r_cnt, r_pr,
        hist, Z, W, bad, total;
};

static CalibLayout make_calib_layout(const sieve_index_view *ix, int64_t nq, int64_t ns,
                                     const sieve_params *p) {
    CalibLayout C{};
    sieve_params wide = *p;
    wide.W = p->nprobe;
    const int64_t nr = nq - ns;
    const Layout a = make_layout(ix, ns, &wide, false), b = make_layout(ix, nr, &wide, false);
    C.inner = a.total >= b.total ? a : b;
    size_t off = C.inner.total;
    auto take = [&](size_t bytes) {
        size_t at = off;
        off += (size_t)round_up((int64_t)std::max<size_t>(bytes, 1), 256);
        return at;
    };
    const int k = p->k, d = ix->d;
    const int words = (int)ceil_div(p->nprobe, 32);
    C.Qs = take((size_t)ns * d * 4);
    C.qs = take((size_t)ns * 8);
    C.s_ids = take((size_t)ns * k * 8);
    C.s_sc = take((size_t)ns * k * 4);
    C.s_cnt = take((size_t)ns * 4);
    C.s_pr = take((size_t)ns * 4);
    C.s_rank = take((size_t)ns * k * 4);
    C.s_hits = take((size_t)ns * words * 4);
    C.rest = take((size_t)nr * 8);
    C.Qr = take((size_t)nr * d * 4);
    C.qr = take((size_t)nr * 8);
    C.r_ids = take((size_t)nr * k * 8);
    C.r_sc = take((size_t)nr * k * 4);
    C.r_cnt = take((size_t)nr * 4);
    C.r_pr = take((size_t)nr * 4);
    C.hist = take((size_t)(p->nprobe + 1) * 8);
    C.Z = take(8);
    C.W = take(4);
    C.bad = take(4);
    C.total = off;
    return C;
}

sieve_status sieve_calibrated_search_workspace_size(const sieve_index_view *ix, int64_t nq,
                                                    int64_t ns, const sieve_params *p,
                                                    size_t *bytes) {
    if (!bytes) return SIEVE_EINVAL;
    sieve_status rc = check_index(ix, true);
    if (rc != SIEVE_OK) return rc;
    if ((rc = check_params(ix, p)) != SIEVE_OK) return rc;
    if (nq < 0 || nq > INT32_MAX / 2 || ns < 0 || ns > nq) return SIEVE_EINVAL;
    const Layout plain = make_layout(ix, nq, p, false);
    *bytes = std::max(plain.total, make_calib_layout(ix, nq, ns, p).total);
    return SIEVE_OK;
}

sieve_status sieve_calibrated_search(const sieve_index_view *ix, const float *Q, int64_t nq,
                                     const int64_t *query_ids, const sieve_params *p,
                                     const int64_t *sample, int64_t ns, double eps,
                                     int64_t min_queries, int32_t fallback_W, int64_t *out_ids,
                                     float *out_scores, int32_t *out_count, int32_t *out_probes,
                                     int32_t *W_out, int64_t *hist_out, int64_t *Z_out, void *ws,
                                     size_t ws_bytes, void *stream) {
    sieve_status rc = check_search(ix, Q, nq, nullptr, p, out_ids, out_scores, out_count, out_probes);
    if (rc != SIEVE_OK) return rc;
    if (!W_out || ns < 0 || ns > nq || (ns > 0 && !sample) || fallback_W < 1 || !(eps == eps) ||
        p->profile || (nq > 0 && !aligned16(Q)) || !ix->centroids)
        return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned char *w = static_cast<unsigned char *>(ws);
    if (hist_out)
        for (int i = 0; i <= p->nprobe; ++i) hist_out[i] = 0;
    if (Z_out) *Z_out = 0;
    if (nq == 0) {
        *W_out = fallback_W;
        return SIEVE_OK;
    }
    if (nq < min_queries || ns == 0) {   // small calls: the fallback window, no sample
        *W_out = fallback_W;
        sieve_params q = *p;
        q.W = fallback_W;
        const Layout L = make_layout(ix, nq, &q, false);
        if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < L.total)
            return SIEVE_EWORKSPACE;
        return search_device(ix, Q, nq, query_ids, nullptr, &q, out_ids, out_scores, out_count,
                             out_probes, nullptr, w, L, st);
    }
    const CalibLayout C = make_calib_layout(ix, nq, ns, p);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < C.total)
        return SIEVE_EWORKSPACE;
    const int k = p->k, d = ix->d;
    const int64_t nr = nq - ns;
    auto F = [&](size_t off) { return reinterpret_cast<float *>(w + off); };
    auto I64 = [&](size_t off) { return reinterpret_cast<int64_t *>(w + off); };
    auto I32 = [&](size_t off) { return reinterpret_cast<int32_t *>(w + off); };
    int *bad_d = I32(C.bad);
    SIEVE_CUDA(calib_check_sample(sample, ns, nq, bad_d, st));
    // 1. the sample, fully probed, with each kept result's rank and the hit bits
    SIEVE_CUDA(calib_gather(Q, query_ids, d, sample, ns, F(C.Qs), I64(C.qs), st));
    sieve_params full = *p;
    full.W = p->nprobe;
    SearchExtras ex{I32(C.s_rank), reinterpret_cast<uint32_t *>(w + C.s_hits)};
    const Layout Ls = make_layout(ix, ns, &full, false);
    rc = search_device(ix, F(C.Qs), ns, query_ids ? I64(C.qs) : nullptr, nullptr, &full,
                       I64(C.s_ids), F(C.s_sc), I32(C.s_cnt), I32(C.s_pr), nullptr, w, Ls, st, &ex);
    if (rc != SIEVE_OK) return rc;
    // 2. the histogram of required windows and W*
    SIEVE_CUDA(calib_pick(reinterpret_cast<const unsigned *>(w + C.s_hits), (int)ceil_div(p->nprobe, 32),
                          I32(C.s_rank), I32(C.s_cnt), ns, k, p->nprobe, eps, fallback_W,
                          reinterpret_cast<unsigned long long *>(w + C.hist),
                          reinterpret_cast<unsigned long long *>(w + C.Z), I32(C.W), st));
    int32_t w_star = 0, bad = 0;
    SIEVE_CUDA(cudaMemcpyAsync(&w_star, I32(C.W), 4, cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaMemcpyAsync(&bad, bad_d, 4, cudaMemcpyDeviceToHost, st));
    if (hist_out)
        SIEVE_CUDA(cudaMemcpyAsync(hist_out, w + C.hist, (size_t)(p->nprobe + 1) * 8,
                                   cudaMemcpyDeviceToHost, st));
    if (Z_out) SIEVE_CUDA(cudaMemcpyAsync(Z_out, w + C.Z, 8, cudaMemcpyDeviceToHost, st));
    SIEVE_CUDA(cudaStreamSynchronize(st));
    if (bad) return SIEVE_EINVAL;   // the sample was not strictly increasing rows of Q
    *W_out = w_star;
    // 3. the rest of the batch under W*, then every row to its place
    if (nr > 0) {
        SIEVE_CUDA(calib_complement(sample, ns, nq, I64(C.rest), st));
        SIEVE_CUDA(calib_gather(Q, query_ids, d, I64(C.rest), nr, F(C.Qr), I64(C.qr), st));
        sieve_params rest = *p;
        rest.W = w_star;
        const Layout Lr = make_layout(ix, nr, &rest, false);
        rc = search_device(ix, F(C.Qr), nr, query_ids ? I64(C.qr) : nullptr, nullptr, &rest,
                           I64(C.r_ids), F(C.r_sc), I32(C.r_cnt), I32(C.r_pr), nullptr, w, Lr, st);
        if (rc != SIEVE_OK) return rc;
        SIEVE_CUDA(calib_scatter(I64(C.rest), nr, k, reinterpret_cast<const long long *>(I64(C.r_ids)),
                                 F(C.r_sc), I32(C.r_cnt), I32(C.r_pr),
                                 reinterpret_cast<long long *>(out_ids), out_scores, out_count,
                                 out_probes, st));
    }
    SIEVE_CUDA(calib_scatter(sample, ns, k, reinterpret_cast<const long long *>(I64(C.s_ids)), F(C.s_sc),
                             I32(C.s_cnt), I32(C.s_pr), reinterpret_cast<long long *>(out_ids),
                             out_scores, out_count, out_probes, st));
    return SIEVE_OK;
}

// ---------------------------------------------------------------------------
// Sharded search (Sec. 6.1's public-100M layout).  Scratch: the inner
// search's workspace (the largest any shard needs), then the shards' results.
struct ShardLayout {
    Layout inner;
    size_t ids, sc, cnt, pr, total;
};

static sieve_status shard_params(const sieve_params *p, const int32_t *W_per_shard, int s,
                                 sieve_params *out) {
    *out = *p;
    if (W_per_shard) out->W = W_per_shard[s];
    return out->W >= 1 ? SIEVE_OK : SIEVE_EINVAL;
}

static ShardLayout make_shard_layout(const sieve_index_view *shards, int nshards, int64_t nq,
                                     const sieve_params *p, const int32_t *W_per_shard) {
    ShardLayout S{};
    for (int s = 0; s < nshards; ++s) {
        sieve_params ps;
        shard_params(p, W_per_shard, s, &ps);
        const Layout L = make_layout(&shards[s], nq, &ps, false);
        if (L.total > S.inner.total) S.inner = L;
    }
    size_t off = S.inner.total;
    auto take = [&](size_t bytes) {
        size_t at = off;
        off += (size_t)round_up((int64_t)std::max<size_t>(bytes, 1), 256);
        return at;
    };
    S.ids = take((size_t)nshards * nq * p->k * 8);
    S.sc = take((size_t)nshards * nq * p->k * 4);
    S.cnt = take((size_t)nshards * nq * 4);
    S.pr = take((size_t)nshards * nq * 4);
    S.total = off;
    return S;
}

static sieve_status check_shards(const sieve_index_view *shards, int32_t nshards,
                                 const sieve_params *p, const int32_t *W_per_shard) {
    if (!shards || nshards < 1) return SIEVE_EINVAL;
    for (int s = 0; s < nshards; ++s) {
        sieve_status rc = check_index(&shards[s], true);
        if (rc != SIEVE_OK) return rc;
        if (shards[s].d != shards[0].d) return SIEVE_EINVAL;
        sieve_params ps;
        if ((rc = shard_params(p, W_per_shard, s, &ps)) != SIEVE_OK) return rc;
        if ((rc = check_params(&shards[s], &ps)) != SIEVE_OK) return rc;
    }
    return SIEVE_OK;
}

sieve_status sieve_sharded_search_workspace_size(const sieve_index_view *shards, int32_t nshards,
                                                 int64_t nq, const sieve_params *p,
                                                 const int32_t *W_per_shard, size_t *bytes) {
    if (!bytes || !p) return SIEVE_EINVAL;
    sieve_status rc = check_shards(shards, nshards, p, W_per_shard);
    if (rc != SIEVE_OK) return rc;
    if (nq < 0 || nq > INT32_MAX / 2) return SIEVE_EINVAL;
    *bytes = make_shard_layout(shards, nshards, nq, p, W_per_shard).total;
    return SIEVE_OK;
}

sieve_status sieve_sharded_search(const sieve_index_view *shards, int32_t nshards, const float *Q,
                                  int64_t nq, const int64_t *query_ids, const sieve_params *p,
                                  const int32_t *W_per_shard, int64_t *out_ids, float *out_scores,
                                  int32_t *out_count, int32_t *out_probes, int32_t *shard_probes,
                                  void *ws, size_t ws_bytes, void *stream) {
    if (!p) return SIEVE_EINVAL;
    sieve_status rc = check_shards(shards, nshards, p, W_per_shard);
    if (rc != SIEVE_OK) return rc;
    if ((rc = check_search(&shards[0], Q, nq, nullptr, p, out_ids, out_scores, out_count,
                           out_probes)) != SIEVE_OK)
        return rc;
    if (p->profile || (nq > 0 && !aligned16(Q))) return SIEVE_EINVAL;
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (nq == 0) return SIEVE_OK;
    const ShardLayout S = make_shard_layout(shards, nshards, nq, p, W_per_shard);
    if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < S.total)
        return SIEVE_EWORKSPACE;
    unsigned char *w = static_cast<unsigned char *>(ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int k = p->k;
    int64_t *ids = reinterpret_cast<int64_t *>(w + S.ids);
    float *sc = reinterpret_cast<float *>(w + S.sc);
    int32_t *cnt = reinterpret_cast<int32_t *>(w + S.cnt);
    int32_t *pr = reinterpret_cast<int32_t *>(w + S.pr);
    for (int s = 0; s < nshards; ++s) {   // each shard ranks and stops on its own
        sieve_params ps;
        shard_params(p, W_per_shard, s, &ps);
        const Layout L = make_layout(&shards[s], nq, &ps, false);
        rc = search_device(&shards[s], Q, nq, query_ids, nullptr, &ps, ids + (int64_t)s * nq * k,
                           sc + (int64_t)s * nq * k, cnt + (int64_t)s * nq, pr + (int64_t)s * nq,
                           nullptr, w, L, st);
        if (rc != SIEVE_OK) return rc;
    }
    SIEVE_CUDA(launch_merge_shards(nshards, nq, k, reinterpret_cast<const long long *>(ids), sc, cnt,
                                   pr, reinterpret_cast<long long *>(out_ids), out_scores, out_count,
                                   out_probes, shard_probes, st));
    return SIEVE_OK;
}

sieve_status sieve_merge_shard_results(int32_t nshards, int64_t nq, int32_t k,
                                       const int64_t *ids, const float *scores,
                                       const int32_t *count, const int32_t *probes,
                                       int64_t *out_ids, float *out_scores, int32_t *out_count,
                                       int32_t *out_probes, int32_t *shard_probes, void *stream) {
    if (nshards < 1 || nq < 0 || k < 1 || k > kMaxK) return SIEVE_EINVAL;
    if (nq > 0 && (!ids || !scores || !count || !probes || !out_ids || !out_scores || !out_count ||
                   !out_probes))
        return SIEVE_EINVAL;
    sieve_status rc = check_device();
    if (rc != SIEVE_OK) return rc;
    SIEVE_CUDA(launch_merge_shards(nshards, nq, k, reinterpret_cast<const long long *>(ids), scores,
                                   count, probes, reinterpret_cast<long long *>(out_ids), out_scores,
                                   out_count, out_probes, shard_probes,
                                   static_cast<cudaStream_t>(stream)));
    return SIEVE_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// sieve_search_noalloc: sieve_search for callers that cannot allocate device
// memory at all (an allocator-free host process, a plug-in running inside a
// host application that owns every allocation, code between a caller's own
// pool resets).  Its scratch is the fixed array below: part of the library
// image, so every GPU that loads the library holds it until the process
// exits, and every call on that GPU shares it.
namespace {

constexpr size_t kNoallocScratchBytes = size_t(64) << 20;   // SIEVE_NOALLOC_SCRATCH_BYTES
static_assert(kNoallocScratchBytes == SIEVE_NOALLOC_SCRATCH_BYTES,
              "the header's scratch size and the array's must agree");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

// Device address of the scratch array on the current device.  In host code
// the array's name is only a host-side stand-in, so the address is asked of
// the runtime, with the device current, on every call: a lookup in the
// loaded module, no allocation.  Nothing is cached, so a context that was
// destroyed and created again (cudaDeviceReset) gets the new address.
sieve_status noalloc_scratch(void **out) {
    void *p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return cuda_fail(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
    *out = p;
    return SIEVE_OK;
}

}  // namespace

extern "C" sieve_status sieve_search_noalloc(const sieve_index_view *ix, const float *Q,
                                             int64_t nq, const int64_t *query_ids,
                                             const int32_t *order, const sieve_params *p,
                                             int64_t *out_ids, float *out_scores,
                                             int32_t *out_count, int32_t *out_probes,
                                             sieve_stats *stats, void *stream) {
    sieve_status rc = check_search(ix, Q, nq, order, p, out_ids, out_scores, out_count, out_probes);
    if (rc != SIEVE_OK) return rc;
    if (nq > 0 && !aligned16(Q)) return SIEVE_EINVAL;
    if (p->profile) return SIEVE_EINVAL;   // event timing is not offered here
    if ((rc = check_device()) != SIEVE_OK) return rc;
    if (stats) std::memset(stats, 0, sizeof(*stats));
    if (nq == 0) return SIEVE_OK;
    const Layout L = make_layout(ix, nq, p, false);
    if (L.total > kNoallocScratchBytes) return SIEVE_ESCRATCH;
    void *ws = nullptr;
    if ((rc = noalloc_scratch(&ws)) != SIEVE_OK) return rc;
    // host-driven rounds: building and instantiating a CUDA graph could
    // allocate, so this entry point never does
    sieve_params hp = *p;
    hp.loop = 1;
    return search_device(ix, Q, nq, query_ids, order, &hp, out_ids, out_scores, out_count,
                         out_probes, stats, static_cast<unsigned char *>(ws), L,
                         static_cast<cudaStream_t>(stream));
}
