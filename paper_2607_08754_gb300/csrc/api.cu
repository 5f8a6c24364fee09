// libslorr C ABI: planning, workspace layout, tensor maps and the launch
// sequence of one regularizer forward + backward (Listing 1, Alg. 2):
//   normcast (or sumsq, cast) -> the T steps' Gram, Poly and Update tiles in
//   one dataflow launch (or 3 T per-phase launches) -> dot -> combine
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <queue>
#include <cstdio>
#include <cstring>
#include <numeric>
#include <string>
#include <vector>

#include "../../include/slorr.h"
#include "internal.h"

using namespace slorr;

namespace {

thread_local std::string g_last_error;

slorr_status fail(slorr_status s, const std::string& msg) {
    g_last_error = msg;
    return s;
}

slorr_status cuda_fail(cudaError_t e, const char* what) {
    g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
    if (e == cudaErrorNoKernelImageForDevice || e == cudaErrorInvalidDeviceFunction)
        return SLORR_ERR_UNSUPPORTED;
    return SLORR_ERR_CUDA;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

void slorr::set_last_error(const std::string& msg) { g_last_error = msg; }

namespace {

struct Geom {
    int m, n, P, Q, Ppad, Qpad, transposed, rows, ld;
    size_t off_x[2], off_a, off_b;
    size_t off_xlo[2], off_alo, off_blo;  // bf16 hi/lo mode: the low parts of X_t, A and M
    size_t off_tf32[10];            // fp32 tensor-core mode: xg[2][2], xu[2][2], a lo, m lo
    int tile_base, tile_count;      // tiles of W (sumsq, dot, combine)
    int xtile_base, xtile_count;    // tiles of the padded iterate (cast, normcast)
};

}  // namespace

struct slorr_handle {
    slorr_options opt;
    std::vector<slorr_shape> shapes;
    std::vector<Geom> geom;
    std::vector<double> coeffs;  // 3 * T
    int elem;                    // Elem of X / A / B
    int esize;
    // item lists (host)
    std::vector<GemmItem> tc_items[3];
    std::vector<GemmItem> simt_items[3];
    std::vector<GemmItem> tf32_items[3];  // fp32 mode on the tensor cores: 128 x 64 tiles
    // dataflow plan: every (step, phase, tile) item, pair by pair
    std::vector<GemmItem> df_items;
    std::vector<int32_t> df_pair_begin;  // df_pairs + 1 offsets into df_items
    std::vector<int32_t> df_seq;         // each df item's rank in the plan's global start order
    int df_pairs = 0;
    double df_makespan = 0.0;            // simulated, in K blocks of a 256 x 256 tile
    double df_work = 0.0;                // total cost / pairs (a lower bound of the makespan)
    double df_chain = 0.0;               // the longest chain of one matrix's phases (the other bound)
    bool df = false;                     // the GEMMs run as the dataflow launch
    std::vector<MemItem> w_items;  // tiles of W (sumsq, dot, combine)
    std::vector<MemItem> x_items;  // tiles of the padded iterate (cast)
    int total_w_tiles = 0;
    int total_x_tiles = 0;
    int total_split_parts = 0;  // 256 x 256 fp32 partial slots of split-K Gram tiles
    int tf32_split_tiles = 0;   // 32 x 32 tiles of the largest padded iterate (fp32 tensor-core mode)
    // workspace layout
    size_t off_status = 0, off_counters = 0, off_scalars = 0, off_partials = 0, off_partials_max = 0,
           off_tilebase = 0, off_tilecount = 0, off_xtilebase = 0, off_xtilecount = 0, off_split_cnt = 0,
           off_split_part = 0, off_mats = 0, off_maps = 0, off_tc_items[3] = {}, off_simt_items[3] = {},
           off_done = 0, off_df_items = 0, off_df_pair_begin = 0, off_coef = 0, off_tf32_mats = 0,
           off_tf32_maps = 0, off_tf32_items[3] = {},
           off_w_items = 0, off_x_items = 0, off_ptrs = 0, off_plan_end = 0, total_bytes = 0;
    // device state
    const void* prepared_ws = nullptr;
    std::vector<const void*> last_ptrs;  // weights then grads last uploaded
    int num_sms = 0;
    // tracing
    bool timing = false;
    std::vector<cudaEvent_t> ev_pool;
    struct Mark { int kind; int kernels; cudaEvent_t start, stop; };
    std::vector<Mark> marks;
    // SLORR_FLAG_GRAPH
    cudaGraphExec_t graph_exec = nullptr;
    std::vector<uintptr_t> graph_key;
    cudaStream_t capture_stream = nullptr;
    ~slorr_handle() {
        if (graph_exec) cudaGraphExecDestroy(graph_exec);
        if (capture_stream) cudaStreamDestroy(capture_stream);
        for (auto& m : marks) {
            cudaEventDestroy(m.start);
            cudaEventDestroy(m.stop);
        }
        for (auto e : ev_pool) cudaEventDestroy(e);
    }
};

namespace {

// Tensor-core GEMM phases as one dataflow launch, or one launch per phase and
// step (build_plan decides; see kDataflowMaxWork).
bool dataflow(const slorr_handle* h) { return h->df; }

// bf16 hi/lo mode (SLORR_COMPUTE_BF16_SPLIT): the iterates, A and M carried
// as bf16 hi and lo parts, every product as three bf16 products.
bool split16(const slorr_handle* h) { return h->opt.compute == SLORR_COMPUTE_BF16_SPLIT; }

bool dataflow_possible(const slorr_handle* h) {
    return h->opt.compute != SLORR_COMPUTE_FP32 && !split16(h) &&
           (h->opt.flags & (SLORR_FLAG_SIMT_GEMM | SLORR_FLAG_PHASE_LAUNCHES)) == 0;
}

// fp32 mode runs its products on the tensor cores as three tf32 products
// (kernels_tf32.cu) unless the CUDA-core kernel is asked for.
bool tf32_tc(const slorr_handle* h) {
    return h->opt.compute == SLORR_COMPUTE_FP32 && (h->opt.flags & SLORR_FLAG_SIMT_GEMM) == 0;
}

// Programmatic dependent launch of the memory passes and the pair kernel.
bool use_pdl(const slorr_handle* h) { return (h->opt.flags & SLORR_FLAG_NO_PDL) == 0; }

// 16-bit iterates on the tensor cores: the norm and the cast share one read of
// W (normcast), and the first Gram and Update epilogues apply the scale.
bool fused_norm(const slorr_handle* h) {
    return h->opt.compute != SLORR_COMPUTE_FP32 &&
           (h->opt.flags & (SLORR_FLAG_SIMT_GEMM | SLORR_FLAG_SEPARATE_NORM)) == 0;
}

constexpr int32_t kKnownFlags = SLORR_FLAG_SIMT_GEMM | SLORR_FLAG_TEST_STALL | SLORR_FLAG_WRITE_GRAD |
                                SLORR_FLAG_NO_PDL | SLORR_FLAG_SEPARATE_NORM | SLORR_FLAG_NO_SPLIT_K |
                                SLORR_FLAG_GRAPH | SLORR_FLAG_PHASE_LAUNCHES | SLORR_FLAG_DATAFLOW;

bool valid_options(const slorr_options& o, std::string* why) {
    if (o.variant != SLORR_HOYER && o.variant != SLORR_NUCLEAR) return *why = "variant", false;
    if (o.compute < SLORR_COMPUTE_FP16 || o.compute > SLORR_COMPUTE_BF16_SPLIT) return *why = "compute", false;
    if (o.dtype != SLORR_F32 && o.dtype != SLORR_BF16) return *why = "dtype", false;
    if (o.iters < 1 || o.iters > kMaxIters) return *why = "iters must be in [1, 16]", false;
    if (!(o.ell > 0.0 && o.ell < 1.0)) return *why = "ell must be in (0, 1)", false;
    if (!(o.safety >= 1.0) || !std::isfinite(o.safety)) return *why = "safety must be >= 1", false;
    if (!std::isfinite(o.cushion) || o.cushion >= 1.0) return *why = "cushion must be < 1", false;
    if (!(o.eps >= 0.f) || !std::isfinite(o.eps)) return *why = "eps must be >= 0", false;
    if (!std::isfinite(o.lambda) || !std::isfinite(o.grad_scale)) return *why = "lambda/grad_scale", false;
    if (!(o.timeout_s > 0.0) || o.timeout_s > 3600.0) return *why = "timeout_s must be in (0, 3600]", false;
    if (o.flags & ~kKnownFlags) return *why = "flags holds a bit this build does not define", false;
    if ((o.flags & SLORR_FLAG_PHASE_LAUNCHES) && (o.flags & SLORR_FLAG_DATAFLOW))
        return *why = "SLORR_FLAG_PHASE_LAUNCHES and SLORR_FLAG_DATAFLOW exclude each other", false;
    if (o.compute == SLORR_COMPUTE_BF16_SPLIT &&
        (o.flags & (SLORR_FLAG_SIMT_GEMM | SLORR_FLAG_SEPARATE_NORM | SLORR_FLAG_DATAFLOW)))
        return *why = "SLORR_COMPUTE_BF16_SPLIT runs on the tensor cores, after the fused norm pass, in per-phase "
                      "launches (no SIMT_GEMM, SEPARATE_NORM or DATAFLOW flag)",
               false;
    return true;
}

// Split K of the CTA-pair kernel's Gram tiles (A = X X^T with K = Qpad).  A
// Gram launch lasts at least as long as its longest tile, and a set with few
// tiles of long K (ResNet-18's 512 x 4608 layers: 3 tiles of K = 4608) leaves
// most pairs idle meanwhile.  The plan assumes 76 pairs (152 SMs): a tile's K
// is split into parts of about max(1024, the launch's K per pair), at most
// kMaxSplit (2) parts.  Each part accumulates its K range; the epilogue warp that
// finishes last adds the parts' fp32 partials in part order.  That warp
// reads every part's 256 x 256 partial, so more parts shorten the main loop
// but lengthen the last epilogue.
constexpr int kPlanPairs = 76;
#ifndef SLORR_SPLIT_MIN_K
#define SLORR_SPLIT_MIN_K 1024
#endif

// Order one phase's items (sorted by cost, largest first) for the pair
// kernel, which hands item i to pair i mod npairs.  Each of kPlanPairs pairs
// keeps the number of items that round-robin gives it; items go to the
// least-loaded pair with room (longest processing time first), then swaps
// between the most-loaded pair and the others lower the largest load.  Pair
// p's j-th item is placed at index j kPlanPairs + p, unless that does not
// lower the largest load of the input order.  Any npairs processes every
// item; kPlanPairs (GB300's 152 SMs as pairs) is the one it balances.
void balance_pairs(std::vector<GemmItem>& v, const std::vector<int64_t>& cost) {
    const int n = kPlanPairs;
    const size_t N = v.size();
    if (N <= size_t(n)) return;
    std::vector<int64_t> rr(n, 0);  // the input order's loads
    for (size_t i = 0; i < N; ++i) rr[i % n] += cost[i];
    std::vector<std::vector<int>> lists(n);
    std::vector<int64_t> load(n, 0);
    std::vector<size_t> cap(n);
    for (int p = 0; p < n; ++p) cap[p] = N / n + (size_t(p) < N % n ? 1 : 0);
    for (size_t i = 0; i < N; ++i) {
        int best = -1;
        for (int p = 0; p < n; ++p)
            if (lists[p].size() < cap[p] && (best < 0 || load[p] < load[best])) best = p;
        lists[best].push_back(int(i));
        load[best] += cost[i];
    }
    // One representative item per distinct cost in a list keeps the search small.
    auto reps = [&](int p) {
        std::vector<int> r;
        for (int i : lists[p]) {
            bool seen = false;
            for (int j : r) seen = seen || cost[j] == cost[i];
            if (!seen) r.push_back(i);
        }
        return r;
    };
    for (int iter = 0; iter < 8 * n; ++iter) {
        const int p = int(std::max_element(load.begin(), load.end()) - load.begin());
        const std::vector<int> rp = reps(p);
        int64_t best_max = load[p];
        int bq = -1, bx = -1, by = -1;
        for (int q = 0; q < n; ++q) {
            if (q == p) continue;
            for (int y : reps(q))
                for (int x : rp) {
                    if (cost[x] <= cost[y]) continue;
                    const int64_t m = std::max(load[p] - cost[x] + cost[y], load[q] - cost[y] + cost[x]);
                    if (m < best_max) best_max = m, bq = q, bx = x, by = y;
                }
        }
        if (bq < 0) break;
        std::replace(lists[p].begin(), lists[p].end(), bx, by);
        std::replace(lists[bq].begin(), lists[bq].end(), by, bx);
        load[p] += cost[by] - cost[bx];
        load[bq] += cost[bx] - cost[by];
    }
    if (*std::max_element(load.begin(), load.end()) >= *std::max_element(rr.begin(), rr.end())) return;
    std::vector<GemmItem> out(N);
    std::vector<char> used(N, 0);
    for (int p = 0; p < n; ++p) {
        std::sort(lists[p].begin(), lists[p].end());  // keep the sorted order within a pair
        for (size_t j = 0; j < lists[p].size(); ++j) {
            const size_t at = j * n + p;
            if (at >= N || used[size_t(lists[p][j])]) return;  // not a permutation: keep the sorted order
            used[size_t(lists[p][j])] = 1;
            out[at] = v[size_t(lists[p][j])];
        }
    }
    v.swap(out);
}

void split_gram_items(slorr_handle* h) {
    h->total_split_parts = 0;
    if (h->opt.compute == SLORR_COMPUTE_FP32 || (h->opt.flags & (SLORR_FLAG_SIMT_GEMM | SLORR_FLAG_NO_SPLIT_K)))
        return;
    std::vector<GemmItem>& items = h->tc_items[kGram];
    double work = 0.0;
    for (const GemmItem& it : items) work += h->geom[it.mat].Qpad;
    const double target = std::max(double(SLORR_SPLIT_MIN_K), work / kPlanPairs);
    std::vector<GemmItem> out;
    for (const GemmItem& it : items) {
        const int K = h->geom[it.mat].Qpad;
        int parts = int(std::ceil(K / target));
        parts = std::min(std::min(parts, kMaxSplit), K / kPairBK);
        if (parts <= 1) {
            out.push_back(it);
            continue;
        }
        for (int q = 0; q < parts; ++q) {
            GemmItem part = it;
            part.ksplit = uint16_t(q | (parts << 8));
            part.sid = uint32_t(h->total_split_parts);
            out.push_back(part);
        }
        h->total_split_parts += parts;
    }
    items.swap(out);
}

// Dataflow plan.  The T steps' Gram, Poly and Update tiles of every matrix
// run in one launch; a matrix's phases are strictly ordered (each phase reads
// what the previous one wrote: Gram X_t -> A, Poly A -> M, Update M, X_t ->
// X_{t+1}), and different matrices are independent.  The items are assigned
// to CTA pairs by list scheduling over a simulated clock: whenever a pair is
// free it takes, among the items whose matrix has finished the previous phase,
// the one with the longest remaining chain of phases below it (the sum, over
// the matrix's remaining phases, of their longest tile plus the latency of a
// dependency), longest tile first among equals.  Each pair runs its items in
// the order of their simulated start times; an item's simulated start is
// later than every start of the items it depends on, so ordering all items by
// start time puts each one after its dependencies, and the earliest item not
// yet finished can always run: the launch cannot deadlock whatever the real
// timings are, provided every pair is resident.
//
// Costs are in K blocks (64) of a 256 x 256 tile: the tile's K blocks, scaled
// by its width (an N = 128 UMMA moves 3/4 of the bytes of an N = 256 one), plus
// one block for its start and epilogue (overlapped with the next tile); Poly
// tiles count 1.6 x (their epilogue reads A and writes M: measured 0.82
// against 1.37 PFLOP/s of MMA work on ViT-L/16-shaped tiles);
// the last part of a split tile adds the parts.  A dependency adds 8 blocks
// (the last increments, the producer's wake-up, the first copies landing;
// 8 measured best on ViT-S, ViT-512 and ViT-B with the 64 KB-stage kernel,
// 12 lengthens ViT-S's chain past the launch-mode threshold).
constexpr double kDepLatency = 8.0;

// Which launch a set gets by default.  Per tile the dataflow launch is a few
// per cent slower than the phase-specialised per-phase kernels (8 epilogue
// warps in every phase, phases and matrices mixed on each pair, a dependency
// hand-off through global memory), and what it saves is the tail of each of
// the 3 T per-phase launches.  Measured on GB300 (bench, one box, both modes
// back to back), it is faster when two things hold:
// - the set is work-bound: its longest chain of one matrix's phases is
//   shorter than the work per pair (chain-bound sets -- ResNet-18 +7%, cfg1
//   +2.6% -- wait on dependency hand-offs instead);
// - the per-phase launches are short: fewer than 7 Gram (or Poly) tiles per
//   pair, so a launch tail is a large share (ViT-S -12%, ViT-512 -7%,
//   ViT-B/16 -4.4%, the 560M decoder's first 4 blocks -4.7%, the first 32 and
//   48 ViT-L/16 matrices -3% and -2%; ViT-B with 24 blocks, 7.6 tiles per
//   pair, +2%; ViT-L/16, 12.6, +3%; 560M, 25.6, +5%).
constexpr double kDataflowMaxChainShare = 0.75;
constexpr double kDataflowMaxRounds = 7.0;

double df_cost(const slorr_handle* h, const GemmItem& it) {
    const Geom& g = h->geom[it.mat];
    const int K = it.phase == kGram ? g.Qpad : g.Ppad;
    int b, e;
    split_range(it, K / 64, &b, &e);
    const double kb = double(e - b) * (0.5 + 0.5 * double(it.nsz) / 256.0);
    double c = (it.phase == kPoly ? 1.6 * kb : kb) + 1.0;
    if (it.ksplit) c += 2.0;
    return c;
}

void build_dataflow(slorr_handle* h, int npairs) {
    h->df_items.clear();
    h->df_seq.clear();
    h->df_pair_begin.assign(size_t(npairs) + 1, 0);
    h->df_pairs = npairs;
    h->df_makespan = 0.0;
    h->df_work = 0.0;
    h->df_chain = 0.0;
    const int count = int(h->shapes.size());
    const int T = h->opt.iters;
    // items of each (matrix, phase), in the per-phase plan's order
    std::vector<std::vector<int>> of(size_t(count) * 3);
    std::vector<double> maxcost(size_t(count) * 3, 0.0);
    for (int ph = 0; ph < 3; ++ph)
        for (size_t i = 0; i < h->tc_items[ph].size(); ++i) {
            const GemmItem& it = h->tc_items[ph][i];
            of[size_t(it.mat) * 3 + ph].push_back(int(i));
            maxcost[size_t(it.mat) * 3 + ph] = std::max(maxcost[size_t(it.mat) * 3 + ph], df_cost(h, it));
        }
    // group g = (mat, t, ph), g = (mat * T + t) * 3 + ph; its successor is g + 1
    // (the matrix's next phase; Update of step t is followed by Gram of t + 1)
    const size_t G = size_t(count) * T * 3;
    auto gmat = [&](size_t g) { return int(g / (size_t(T) * 3)); };
    auto gstep = [&](size_t g) { return int(g / 3 % size_t(T)); };
    auto gph = [&](size_t g) { return int(g % 3); };
    std::vector<double> level(G, 0.0), gend(G, 0.0);
    std::vector<int> left(G, 0);
    std::vector<uint32_t> base(G, 0);
    for (int m = 0; m < count; ++m) {
        double acc = 0.0;
        for (int k = T * 3 - 1; k >= 0; --k) {
            acc += maxcost[size_t(m) * 3 + k % 3] + kDepLatency;
            level[size_t(m) * T * 3 + k] = acc;
        }
        uint32_t done = 0;
        for (int k = 0; k < T * 3; ++k) {
            base[size_t(m) * T * 3 + k] = done;
            left[size_t(m) * T * 3 + k] = int(of[size_t(m) * 3 + k % 3].size());
            done += uint32_t(of[size_t(m) * 3 + k % 3].size()) * kDoneIncPerItem;
        }
    }
    struct Ready {
        double level, cost;
        int mat, order;
        size_t g;
        int src;
        bool operator<(const Ready& o) const {  // max-heap: higher level, then longer, then lower index
            if (level != o.level) return level < o.level;
            if (cost != o.cost) return cost < o.cost;
            if (mat != o.mat) return mat > o.mat;
            return order > o.order;
        }
    };
    std::priority_queue<Ready> ready;
    using TimedGroup = std::pair<double, size_t>;  // (ready time, group)
    std::priority_queue<TimedGroup, std::vector<TimedGroup>, std::greater<TimedGroup>> pending;
    using Free = std::pair<double, int>;  // (free time, pair)
    std::priority_queue<Free, std::vector<Free>, std::greater<Free>> pairs;
    for (int q = 0; q < npairs; ++q) pairs.push({0.0, q});
    auto release = [&](size_t g) {
        const std::vector<int>& v = of[size_t(gmat(g)) * 3 + gph(g)];
        for (size_t k = 0; k < v.size(); ++k) {
            const GemmItem& it = h->tc_items[gph(g)][size_t(v[k])];
            ready.push(Ready{level[g], df_cost(h, it), gmat(g), int(k), g, v[k]});
        }
    };
    // the two lower bounds of the makespan
    for (int m = 0; m < count; ++m) h->df_chain = std::max(h->df_chain, level[size_t(m) * T * 3] - kDepLatency);
    for (int ph = 0; ph < 3; ++ph)
        for (const GemmItem& it : h->tc_items[ph]) h->df_work += T * df_cost(h, it) / npairs;
    // every matrix has at least one tile in every phase, so each group is
    // released when its predecessor's last item is assigned
    size_t total = 0;
    for (int m = 0; m < count; ++m) {
        const size_t g0 = size_t(m) * T * 3;
        for (int k = 0; k < T * 3; ++k) total += size_t(left[g0 + k]);
        pending.push({0.0, g0});
    }
    struct Assigned {
        double start;
        int pair;
        size_t g;
        int src;
    };
    std::vector<Assigned> out;
    out.reserve(total);
    while (out.size() < total) {
        Free f = pairs.top();
        pairs.pop();
        while (!pending.empty() && pending.top().first <= f.first) {
            release(pending.top().second);
            pending.pop();
        }
        if (ready.empty()) {
            if (pending.empty()) break;  // not reachable: every group is released once its predecessor ends
            pairs.push({pending.top().first, f.second});
            continue;
        }
        const Ready r = ready.top();
        ready.pop();
        const double end = f.first + r.cost;
        out.push_back(Assigned{f.first, f.second, r.g, r.src});
        gend[r.g] = std::max(gend[r.g], end);
        h->df_makespan = std::max(h->df_makespan, end);
        // the matrix's next (step, phase) becomes ready when this one ends
        if (--left[r.g] == 0 && r.g % (size_t(T) * 3) + 1 < size_t(T) * 3)
            pending.push({gend[r.g] + kDepLatency, r.g + 1});
        pairs.push({end, f.second});
    }
    // global order: by simulated start, then pair
    std::vector<size_t> order(out.size());
    std::iota(order.begin(), order.end(), size_t(0));
    std::stable_sort(order.begin(), order.end(), [&](size_t a, size_t b) {
        if (out[a].start != out[b].start) return out[a].start < out[b].start;
        return out[a].pair < out[b].pair;
    });
    std::vector<int32_t> rank(out.size());
    for (size_t k = 0; k < order.size(); ++k) rank[order[k]] = int32_t(k);
    // pair-major layout; each pair's items are already in start order
    std::vector<std::vector<size_t>> per(static_cast<size_t>(npairs));
    for (size_t k = 0; k < out.size(); ++k) per[size_t(out[k].pair)].push_back(k);
    for (int q = 0; q < npairs; ++q) {
        h->df_pair_begin[size_t(q)] = int32_t(h->df_items.size());
        for (size_t k : per[size_t(q)]) {
            const Assigned& a = out[k];
            GemmItem it = h->tc_items[gph(a.g)][size_t(a.src)];
            it.step = uint8_t(gstep(a.g));
            it.phase = uint8_t(gph(a.g));
            it.wait = base[a.g];
            h->df_items.push_back(it);
            h->df_seq.push_back(rank[k]);
        }
    }
    h->df_pair_begin[size_t(npairs)] = int32_t(h->df_items.size());
}

void build_plan(slorr_handle* h) {
    const int count = int(h->shapes.size());
    h->geom.resize(count);
    for (int i = 0; i < 3; ++i) {
        h->tc_items[i].clear();
        h->simt_items[i].clear();
        h->tf32_items[i].clear();
    }
    h->w_items.clear();
    h->x_items.clear();
    int tile_base = 0, xtile_base = 0;
    for (int i = 0; i < count; ++i) {
        Geom& g = h->geom[i];
        g.m = int(h->shapes[i].m);
        g.n = int(h->shapes[i].n);
        g.transposed = g.m > g.n ? 1 : 0;
        g.P = std::min(g.m, g.n);
        g.Q = std::max(g.m, g.n);
        g.Ppad = int(align_up(size_t(g.P), kPadRows));
        g.Qpad = int(align_up(size_t(g.Q), kPadCols));
        // iterate buffer in W's orientation
        g.rows = g.transposed ? g.Qpad : g.Ppad;
        g.ld = g.transposed ? g.Ppad : g.Qpad;
        // memory-pass tiles: kMemRows x kMemCols of the matrix (of the padded
        // iterate buffer for the cast), or, when the rows are a multiple of 128
        // elements (then ld == n), runs of that many consecutive elements
        const bool flat = g.ld == g.n;
        constexpr int64_t kTileElems = int64_t(kMemRows) * kMemCols;
        g.tile_base = tile_base;
        g.xtile_base = xtile_base;
        int seq = 0, xseq = 0;
        if (flat) {
            const int64_t wt = (int64_t(g.m) * g.n + kTileElems - 1) / kTileElems;
            const int64_t xt = (int64_t(g.rows) * g.ld + kTileElems - 1) / kTileElems;
            for (int64_t t = 0; t < wt && t <= 65535; ++t)
                h->w_items.push_back(MemItem{uint16_t(i), kFlatTile, 0, uint16_t(seq++)});
            for (int64_t t = 0; t < xt && t <= 65535; ++t)
                h->x_items.push_back(MemItem{uint16_t(i), kFlatTile, 0, uint16_t(xseq++)});
            if (wt > 65535 || xt > 65535) seq = xseq = 65536;  // rejected by slorr_create
        } else {
            const int tr = (g.m + kMemRows - 1) / kMemRows, tc = (g.n + kMemCols - 1) / kMemCols;
            for (int r = 0; r < tr; ++r)
                for (int c = 0; c < tc; ++c)
                    h->w_items.push_back(MemItem{uint16_t(i), uint16_t(r), uint16_t(c), uint16_t(seq++)});
            for (int r = 0; r < (g.rows + kMemRows - 1) / kMemRows; ++r)
                for (int c = 0; c < (g.ld + kMemCols - 1) / kMemCols; ++c)
                    h->x_items.push_back(MemItem{uint16_t(i), uint16_t(r), uint16_t(c), uint16_t(xseq++)});
        }
        g.tile_count = seq;
        g.xtile_count = xseq;
        tile_base += seq;
        xtile_base += xseq;
        // tensor-core tiles: msz x nsz with msz, nsz <= 256.  The Gram and
        // Poly outputs are symmetric: tiles lying strictly below the diagonal
        // (in 128 x 128 blocks) are skipped, and their readers take those
        // blocks MN-major from the stored transpose.
        for (int ph = 0; ph < 3; ++ph) {
            const int N = ph == kUpdate ? g.Qpad : g.Ppad;
            for (int tm = 0; tm * 256 < g.Ppad; ++tm) {
                const int msz = std::min(256, g.Ppad - tm * 256);
                for (int tn = 0; tn * 256 < N; ++tn) {
                    const int nsz = std::min(256, N - tn * 256);
                    if (ph != kUpdate && (2 * tn + nsz / 128 - 1) < tm * 2) continue;
                    h->tc_items[ph].push_back(
                        GemmItem{uint16_t(i), uint16_t(tm), uint16_t(tn), uint16_t(nsz), uint16_t(msz), 0});
                    h->tc_items[ph].back().phase = uint8_t(ph);
                }
            }
            // fp32 tensor-core tiles (128 x 64); the symmetric Gram and Poly keep
            // those that reach the diagonal
            if (tf32_tc(h))
                for (int tm = 0; tm < g.Ppad / 128; ++tm)
                    for (int tn = 0; tn < N / 64; ++tn) {
                        if (ph != kUpdate && (tn + 1) * 64 <= tm * 128) continue;
                        h->tf32_items[ph].push_back(GemmItem{uint16_t(i), uint16_t(tm), uint16_t(tn), 64, 128, 0});
                        h->tf32_items[ph].back().phase = uint8_t(ph);
                    }
            // CUDA-core tiles; the symmetric Gram and Poly keep those on or above the diagonal
            for (int tm = 0; tm < g.Ppad / kSimtTile; ++tm)
                for (int tn = (ph == kUpdate ? 0 : tm); tn < N / kSimtTile; ++tn) {
                    h->simt_items[ph].push_back(
                        GemmItem{uint16_t(i), uint16_t(tm), uint16_t(tn), kSimtTile, kSimtTile, 0});
                    h->simt_items[ph].back().phase = uint8_t(ph);
                }
        }
    }
    h->total_w_tiles = tile_base;
    h->total_x_tiles = xtile_base;
    h->tf32_split_tiles = 0;
    if (tf32_tc(h))
        for (const Geom& g : h->geom) h->tf32_split_tiles = std::max(h->tf32_split_tiles, (g.Ppad / 32) * (g.Qpad / 32));
    split_gram_items(h);
    // Longest K first (stable: keeps a matrix's tiles together).
    for (int ph = 0; ph < 3; ++ph) {
        auto kdim = [&](const GemmItem& it) {
            const Geom& g = h->geom[it.mat];
            const int K = ph == kGram ? g.Qpad : g.Ppad;
            int b, e;
            split_range(it, K / kPairBK, &b, &e);
            return it.ksplit ? (e - b) * kPairBK : K;
        };
        std::stable_sort(h->tc_items[ph].begin(), h->tc_items[ph].end(),
                         [&](const GemmItem& a, const GemmItem& b) { return kdim(a) > kdim(b); });
        // Balance the pairs' total K (plus one K block per tile for its
        // fixed cost).  For ViT-L/16's Gram tiles (K = 4096, 3072, 1024) the
        // largest total drops from 40960 to 38912 (ideal 38804); the Gram
        // launches take 1.7% less time than in plain sorted order.
        std::vector<int64_t> cost;
        for (const GemmItem& it : h->tc_items[ph]) cost.push_back(kdim(it) + 64);
        balance_pairs(h->tc_items[ph], cost);
    }
    // the dataflow plan for GB300's 76 pairs (prepare() re-plans for a device
    // that holds another number of pairs at once), kept for sets below the
    // measured crossover or when asked for
    h->df = false;
    if (dataflow_possible(h)) {
        build_dataflow(h, kPlanPairs);
        const double rounds = double(std::min(h->tc_items[kGram].size(), h->tc_items[kPoly].size())) / kPlanPairs;
        h->df = (h->opt.flags & SLORR_FLAG_DATAFLOW) ||
                (h->df_chain < kDataflowMaxChainShare * h->df_work && rounds < kDataflowMaxRounds);
        if (!h->df) {
            h->df_items.clear();
            h->df_seq.clear();
            h->df_pair_begin.clear();
            h->df_pairs = 0;
        }
    }

    // Workspace layout.
    size_t off = 0;
    h->off_status = off;
    off += 256;
    h->off_counters = off;
    off += size_t(count + 1) * 4;
    h->off_done = off;  // zeroed together with the counters at the start of each call
    off = align_up(off + size_t(count) * 4, 256);
    h->off_scalars = off;
    off = align_up(off + size_t(count) * sizeof(MatScalars), 256);
    h->off_partials = off;
    off = align_up(off + size_t(std::max(h->total_w_tiles, h->total_x_tiles)) * 4, 256);
    h->off_partials_max = off;
    off = align_up(off + size_t(h->total_x_tiles) * 4, 256);
    h->off_split_cnt = off;
    off = align_up(off + size_t(h->total_split_parts) * 16 * 4, 256);
    h->off_tilebase = off;
    off = align_up(off + size_t(count) * 4, 256);
    h->off_tilecount = off;
    off = align_up(off + size_t(count) * 4, 256);
    h->off_xtilebase = off;
    off = align_up(off + size_t(count) * 4, 256);
    h->off_xtilecount = off;
    off = align_up(off + size_t(count) * 4, 256);
    h->off_mats = off;
    off = align_up(off + size_t(count) * sizeof(MatDev), 256);
    h->off_maps = off;
    off = align_up(off + size_t(count) * kMapsPerMatrix * 128, 256);
    for (int ph = 0; ph < 3; ++ph) {
        h->off_tc_items[ph] = off;
        off = align_up(off + h->tc_items[ph].size() * sizeof(GemmItem), 256);
        h->off_simt_items[ph] = off;
        off = align_up(off + h->simt_items[ph].size() * sizeof(GemmItem), 256);
    }
    for (int ph = 0; ph < 3; ++ph) {
        h->off_tf32_items[ph] = off;
        off = align_up(off + h->tf32_items[ph].size() * sizeof(GemmItem), 256);
    }
    const bool tf32 = tf32_tc(h);
    h->off_tf32_mats = off;
    off = align_up(off + (tf32 ? size_t(count) * sizeof(MatTf32) : 0), 256);
    h->off_tf32_maps = off;
    off = align_up(off + (tf32 ? size_t(count) * kTf32MapsPerMatrix * 128 : 0), 256);
    h->off_coef = off;
    off = align_up(off + size_t(3 * h->opt.iters) * sizeof(float), 256);
    h->off_df_items = off;
    off = align_up(off + h->df_items.size() * sizeof(GemmItem), 256);
    h->off_df_pair_begin = off;
    off = align_up(off + size_t(dataflow(h) ? kMaxPlanPairs + 1 : 0) * 4, 256);
    h->off_w_items = off;
    off = align_up(off + h->w_items.size() * sizeof(MemItem), 256);
    h->off_x_items = off;
    off = align_up(off + h->x_items.size() * sizeof(MemItem), 256);
    h->off_ptrs = off;
    off = align_up(off + size_t(2 * count) * sizeof(void*), 1024);
    h->off_plan_end = off;
    h->off_split_part = off;
    off = align_up(off + size_t(h->total_split_parts) * 65536 * 4, 1024);
    for (int i = 0; i < count; ++i) {
        Geom& g = h->geom[i];
        const size_t xbytes = size_t(g.rows) * g.ld * h->esize;
        const size_t pbytes = size_t(g.Ppad) * g.Ppad * h->esize;
        g.off_x[0] = off;
        off = align_up(off + xbytes, 1024);
        g.off_x[1] = off;
        off = align_up(off + xbytes, 1024);
        g.off_a = off;
        off = align_up(off + pbytes, 1024);
        g.off_b = off;
        off = align_up(off + pbytes, 1024);
        g.off_xlo[0] = g.off_xlo[1] = g.off_alo = g.off_blo = 0;
        if (split16(h)) {
            g.off_xlo[0] = off;
            off = align_up(off + xbytes, 1024);
            g.off_xlo[1] = off;
            off = align_up(off + xbytes, 1024);
            g.off_alo = off;
            off = align_up(off + pbytes, 1024);
            g.off_blo = off;
            off = align_up(off + pbytes, 1024);
        }
        if (tf32) {
            // xg[b][h] (Ppad x Qpad) and xu[b][h] (Qpad x Ppad), then the lo halves of A and M
            for (int k = 0; k < 8; ++k) {
                g.off_tf32[k] = off;
                off = align_up(off + size_t(g.Ppad) * g.Qpad * 4, 1024);
            }
            for (int k = 8; k < 10; ++k) {
                g.off_tf32[k] = off;
                off = align_up(off + pbytes, 1024);
            }
        }
    }
    h->total_bytes = off;
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// Row-major rows x cols 16-bit matrix seen as a 3-D tensor of 64-element
// chunks: x = the element within a chunk, y = the row, z = the chunk along
// the row (128 bytes apart).  One box is 128 rows of two chunks (32 KB,
// 128-byte swizzle): the K-major half of a CTA-pair operand (rows MN, chunks
// K) or its MN-major half (rows K, chunks MN) for a 128-wide K block.
bool encode_map(CUtensorMap* map, void* base, int rows, int cols, bool bf16) {
    auto enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[3] = {64u, cuuint64_t(rows), cuuint64_t(cols / 64)};
    cuuint64_t strides[2] = {cuuint64_t(cols) * 2, 128u};
    cuuint32_t box[3] = {64u, 128u, cuuint32_t(kPairBK / 64)};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, base,
                     dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Row-major rows x cols fp32 matrix read by the fp32 tensor-core kernel in
// boxes of 32 (contiguous, 128 bytes, 128-byte swizzle) x 64 rows.
bool encode_map_f32(CUtensorMap* map, void* base, int rows, int cols) {
    auto enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {cuuint64_t(cols), cuuint64_t(rows)};
    cuuint64_t strides[1] = {cuuint64_t(cols) * 4};
    cuuint32_t box[2] = {32, 64};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <typename T>
void put(std::vector<uint8_t>& buf, size_t off, const T* src, size_t n) {
    if (n) std::memcpy(buf.data() + off, src, n * sizeof(T));
}

slorr_status prepare(slorr_handle* h, uint8_t* ws, cudaStream_t st) {
    if (h->prepared_ws == ws) return SLORR_OK;
    const int count = int(h->shapes.size());
    if (h->num_sms == 0) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return cuda_fail(e, "device query");
    }
    if (dataflow(h)) {
        // every pair of the dataflow launch must be resident at once: plan for
        // as many pairs as this device holds (76 on a GB300)
        int cap = 0;
        cudaError_t e = tc_pair_dataflow_capacity(h->elem, h->num_sms, &cap);
        if (e != cudaSuccess) return cuda_fail(e, "occupancy query");
        const int npairs = std::min(std::min(cap, h->num_sms / 2), kMaxPlanPairs);
        if (npairs < 1) return fail(SLORR_ERR_UNSUPPORTED, "no CTA pair of the tensor-core kernel fits this device");
        if (npairs != h->df_pairs) build_dataflow(h, npairs);
    }
    std::vector<uint8_t> plan(h->off_plan_end - h->off_tilebase, 0);
    const size_t base = h->off_tilebase;
    std::vector<int32_t> tb(count), tcnt(count), xtb(count), xtcnt(count);
    std::vector<MatDev> mats(count);
    std::vector<uint8_t> maps(size_t(count) * kMapsPerMatrix * 128, 0);
    const bool tf32 = tf32_tc(h);
    std::vector<MatTf32> tmats(tf32 ? size_t(count) : 0);
    std::vector<uint8_t> tmaps(tf32 ? size_t(count) * kTf32MapsPerMatrix * 128 : 0, 0);
    const bool tc = h->opt.compute != SLORR_COMPUTE_FP32;
    for (int i = 0; i < count; ++i) {
        const Geom& g = h->geom[i];
        tb[i] = g.tile_base;
        tcnt[i] = g.tile_count;
        xtb[i] = g.xtile_base;
        xtcnt[i] = g.xtile_count;
        MatDev& md = mats[i];
        md.x[0] = ws + g.off_x[0];
        md.x[1] = ws + g.off_x[1];
        md.a = ws + g.off_a;
        md.b = ws + g.off_b;
        const bool lo = split16(h);
        md.xlo[0] = lo ? ws + g.off_xlo[0] : nullptr;
        md.xlo[1] = lo ? ws + g.off_xlo[1] : nullptr;
        md.alo = lo ? ws + g.off_alo : nullptr;
        md.blo = lo ? ws + g.off_blo : nullptr;
        md.m = g.m;
        md.n = g.n;
        md.P = g.P;
        md.Q = g.Q;
        md.Ppad = g.Ppad;
        md.Qpad = g.Qpad;
        md.transposed = g.transposed;
        md.rows = g.rows;
        md.ld = g.ld;
        md.pad_ = 0;
        if (tc) {
            const bool bf = h->opt.compute == SLORR_COMPUTE_BF16 || lo;
            CUtensorMap* mp = reinterpret_cast<CUtensorMap*>(maps.data() + size_t(i) * kMapsPerMatrix * 128);
            bool ok = true;
            for (int b = 0; b < 2; ++b) ok = ok && encode_map(mp + b, md.x[b], g.rows, g.ld, bf);
            ok = ok && encode_map(mp + 2, md.a, g.Ppad, g.Ppad, bf);
            ok = ok && encode_map(mp + 3, md.b, g.Ppad, g.Ppad, bf);
            if (lo) {
                for (int b = 0; b < 2; ++b) ok = ok && encode_map(mp + 4 + b, md.xlo[b], g.rows, g.ld, true);
                ok = ok && encode_map(mp + 6, md.blo, g.Ppad, g.Ppad, true);
                ok = ok && encode_map(mp + 7, md.alo, g.Ppad, g.Ppad, true);
            }
            if (!ok) return fail(SLORR_ERR_CUDA, "cuTensorMapEncodeTiled failed");
        }
        if (tf32) {
            MatTf32& mt = tmats[i];
            for (int b = 0; b < 2; ++b)
                for (int hl = 0; hl < 2; ++hl) {
                    mt.xg[b][hl] = ws + g.off_tf32[2 * b + hl];
                    mt.xu[b][hl] = ws + g.off_tf32[4 + 2 * b + hl];
                }
            mt.a[0] = md.a;
            mt.a[1] = ws + g.off_tf32[8];
            mt.m[0] = md.b;
            mt.m[1] = ws + g.off_tf32[9];
            CUtensorMap* mp = reinterpret_cast<CUtensorMap*>(tmaps.data() + size_t(i) * kTf32MapsPerMatrix * 128);
            bool ok = true;
            for (int b = 0; b < 2; ++b)
                for (int hl = 0; hl < 2; ++hl) {
                    ok = ok && encode_map_f32(mp + 2 * b + hl, mt.xg[b][hl], g.Ppad, g.Qpad);
                    ok = ok && encode_map_f32(mp + 4 + 2 * b + hl, mt.xu[b][hl], g.Qpad, g.Ppad);
                }
            for (int hl = 0; hl < 2; ++hl) {
                ok = ok && encode_map_f32(mp + 8 + hl, mt.a[hl], g.Ppad, g.Ppad);
                ok = ok && encode_map_f32(mp + 10 + hl, mt.m[hl], g.Ppad, g.Ppad);
            }
            if (!ok) return fail(SLORR_ERR_CUDA, "cuTensorMapEncodeTiled failed (fp32 operands)");
        }
    }
    put(plan, h->off_tilebase - base, tb.data(), tb.size());
    put(plan, h->off_tilecount - base, tcnt.data(), tcnt.size());
    put(plan, h->off_xtilebase - base, xtb.data(), xtb.size());
    put(plan, h->off_xtilecount - base, xtcnt.data(), xtcnt.size());
    put(plan, h->off_mats - base, mats.data(), mats.size());
    put(plan, h->off_maps - base, maps.data(), maps.size());
    put(plan, h->off_tf32_mats - base, tmats.data(), tmats.size());
    put(plan, h->off_tf32_maps - base, tmaps.data(), tmaps.size());
    for (int ph = 0; ph < 3; ++ph) {
        put(plan, h->off_tc_items[ph] - base, h->tc_items[ph].data(), h->tc_items[ph].size());
        put(plan, h->off_simt_items[ph] - base, h->simt_items[ph].data(), h->simt_items[ph].size());
        put(plan, h->off_tf32_items[ph] - base, h->tf32_items[ph].data(), h->tf32_items[ph].size());
    }
    std::vector<float> coef(h->coeffs.begin(), h->coeffs.end());
    put(plan, h->off_coef - base, coef.data(), coef.size());
    put(plan, h->off_df_items - base, h->df_items.data(), h->df_items.size());
    put(plan, h->off_df_pair_begin - base, h->df_pair_begin.data(), h->df_pair_begin.size());
    put(plan, h->off_w_items - base, h->w_items.data(), h->w_items.size());
    put(plan, h->off_x_items - base, h->x_items.data(), h->x_items.size());
    cudaError_t e = cudaMemcpyAsync(ws + base, plan.data(), plan.size(), cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(ws + h->off_status, 0, h->off_tilebase - h->off_status, st);
    if (e != cudaSuccess) return cuda_fail(e, "plan upload");
    h->prepared_ws = ws;
    h->last_ptrs.clear();
    return SLORR_OK;
}

slorr_status upload_ptrs(slorr_handle* h, uint8_t* ws, const void* const* weights, void* const* grads,
                         cudaStream_t st) {
    const int count = int(h->shapes.size());
    std::vector<const void*> ptrs(size_t(2 * count));
    for (int i = 0; i < count; ++i) {
        ptrs[i] = weights[i];
        ptrs[count + i] = grads ? grads[i] : nullptr;
    }
    if (ptrs == h->last_ptrs) return SLORR_OK;
    cudaError_t e = cudaMemcpyAsync(ws + h->off_ptrs, ptrs.data(), ptrs.size() * sizeof(void*),
                                    cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, "pointer upload");
    h->last_ptrs = ptrs;
    return SLORR_OK;
}

cudaEvent_t take_event(slorr_handle* h) {
    if (!h->ev_pool.empty()) {
        cudaEvent_t e = h->ev_pool.back();
        h->ev_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

// Brackets one launch with events when tracing is on.
struct Traced {
    slorr_handle* h;
    cudaStream_t st;
    int kind;
    cudaEvent_t start = nullptr;
    Traced(slorr_handle* h_, int kind_, cudaStream_t st_) : h(h_), st(st_), kind(kind_) {
        if (h->timing && (start = take_event(h)) != nullptr) cudaEventRecord(start, st);
    }
    void done(int kernels = 1) {
        if (!start) return;
        cudaEvent_t stop = take_event(h);
        if (!stop) {
            h->ev_pool.push_back(start);
            return;
        }
        cudaEventRecord(stop, st);
        h->marks.push_back({kind, kernels, start, stop});
        start = nullptr;
    }
};

slorr_status check_matrix_ptrs(const slorr_handle* h, const void* const* arr, const char* what) {
    if (!arr) return fail(SLORR_ERR_INVALID_ARG, std::string(what) + " array is NULL");
    for (size_t i = 0; i < h->shapes.size(); ++i) {
        if (!arr[i]) return fail(SLORR_ERR_INVALID_ARG, std::string(what) + " pointer is NULL");
        if (reinterpret_cast<uintptr_t>(arr[i]) % 16 != 0)
            return fail(SLORR_ERR_INVALID_ARG, std::string(what) + " pointer is not 16-byte aligned");
    }
    return SLORR_OK;
}

MemLaunch mem_params(slorr_handle* h, uint8_t* ws, float* loss, float* per, int cur) {
    MemLaunch p{};
    p.mats = reinterpret_cast<const MatDev*>(ws + h->off_mats);
    p.scalars = reinterpret_cast<MatScalars*>(ws + h->off_scalars);
    p.partials = reinterpret_cast<float*>(ws + h->off_partials);
    p.partials_max = reinterpret_cast<float*>(ws + h->off_partials_max);
    p.tile_base = reinterpret_cast<const int32_t*>(ws + h->off_tilebase);
    p.tile_count = reinterpret_cast<const int32_t*>(ws + h->off_tilecount);
    p.counters = reinterpret_cast<uint32_t*>(ws + h->off_counters);
    p.status = reinterpret_cast<uint32_t*>(ws + h->off_status);
    p.count = int(h->shapes.size());
    p.cur = cur;
    p.elem = h->elem;
    p.wdtype = h->opt.dtype == SLORR_BF16 ? 1 : 0;
    p.variant = h->opt.variant;
    p.out_mode = (h->opt.flags & SLORR_FLAG_WRITE_GRAD) ? kOutOverwrite : kOutAccumulate;
    p.pdl = use_pdl(h) ? 1 : 0;
    p.eps = h->opt.eps;
    p.lambda = h->opt.lambda;
    p.grad_scale = h->opt.grad_scale;
    p.loss_out = loss;
    p.per_matrix_out = per;
    p.weights = reinterpret_cast<const void* const*>(ws + h->off_ptrs);
    p.grads = reinterpret_cast<void* const*>(ws + h->off_ptrs + h->shapes.size() * sizeof(void*));
    return p;
}

// descent: grads is NULL and the combine pass applies W -= eta * lambda *
// grad_scale * G in place (the weights are then written, through a non-const
// pointer the caller gave slorr_reg_descent_step).
slorr_status launch_all(slorr_handle* h, uint8_t* ws, float* loss, float* per, int steps, bool finish,
                        cudaStream_t st, bool descent, float eta);

// SLORR_FLAG_GRAPH: the call's launches are captured once into a CUDA graph
// and replayed while the workspace, the loss and value outputs, T and eta
// stay the same (the weight and gradient pointers live in the workspace, so
// new tensors need no new graph).  A stream that is already being captured
// gets the launches themselves.
slorr_status launch_graph(slorr_handle* h, uint8_t* ws, float* loss, float* per, int steps, cudaStream_t st,
                          bool descent, float eta) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(st, &cs);
    if (e != cudaSuccess) return cuda_fail(e, "stream query");
    if (cs != cudaStreamCaptureStatusNone) return launch_all(h, ws, loss, per, steps, true, st, descent, eta);
    uint32_t eta_bits = 0;
    std::memcpy(&eta_bits, &eta, 4);
    const std::vector<uintptr_t> key = {reinterpret_cast<uintptr_t>(ws), reinterpret_cast<uintptr_t>(loss),
                                        reinterpret_cast<uintptr_t>(per), uintptr_t(steps), uintptr_t(descent),
                                        uintptr_t(eta_bits)};
    if (h->graph_exec == nullptr || key != h->graph_key) {
        if (h->graph_exec != nullptr) {
            cudaGraphExecDestroy(h->graph_exec);
            h->graph_exec = nullptr;
        }
        // relaxed: the first launch of each kernel configuration queries its
        // occupancy, which the stricter capture modes forbid
        // captured on a stream of the handle's own (the caller's may be the
        // legacy default stream, which cannot be captured); launched on st
        if (h->capture_stream == nullptr) {
            e = cudaStreamCreateWithFlags(&h->capture_stream, cudaStreamNonBlocking);
            if (e != cudaSuccess) {
                h->capture_stream = nullptr;
                return cuda_fail(e, "capture stream");
            }
        }
        cudaStream_t cap = h->capture_stream;
        e = cudaStreamBeginCapture(cap, cudaStreamCaptureModeRelaxed);
        if (e != cudaSuccess) return cuda_fail(e, "graph capture");
        const slorr_status s = launch_all(h, ws, loss, per, steps, true, cap, descent, eta);
        cudaGraph_t graph = nullptr;
        e = cudaStreamEndCapture(cap, &graph);
        if (s != SLORR_OK) {
            if (graph) cudaGraphDestroy(graph);
            return s;
        }
        if (e != cudaSuccess) return cuda_fail(e, "graph capture");
        e = cudaGraphInstantiate(&h->graph_exec, graph, 0);
        cudaGraphDestroy(graph);
        if (e != cudaSuccess) {
            h->graph_exec = nullptr;
            return cuda_fail(e, "graph instantiation");
        }
        h->graph_key = key;
    }
    e = cudaGraphLaunch(h->graph_exec, st);
    if (e != cudaSuccess) return cuda_fail(e, "graph launch");
    return SLORR_OK;
}

slorr_status run(slorr_handle* h, const void* const* weights, void* const* grads, float* loss, float* per,
                 void* workspace, size_t ws_bytes, int steps, bool finish, cudaStream_t st,
                 bool descent = false, float eta = 0.f) {
    if (!h) return fail(SLORR_ERR_INVALID_ARG, "handle is NULL");
    slorr_status s = check_matrix_ptrs(h, weights, "weight");
    if (s != SLORR_OK) return s;
    if (descent) {
        if (!std::isfinite(eta)) return fail(SLORR_ERR_INVALID_ARG, "eta must be finite");
        if (!std::isfinite(eta * h->opt.lambda * h->opt.grad_scale))
            return fail(SLORR_ERR_INVALID_ARG, "eta * lambda * grad_scale overflows");
        grads = const_cast<void* const*>(weights);
    }
    if (finish) {
        if (!loss) return fail(SLORR_ERR_INVALID_ARG, "loss_out is NULL");
        if (!descent) {
            s = check_matrix_ptrs(h, grads, "grad");
            if (s != SLORR_OK) return s;
            for (size_t i = 0; i < h->shapes.size(); ++i)
                if (grads[i] == weights[i]) return fail(SLORR_ERR_INVALID_ARG, "a grad aliases its weight");
        }
    }
    if (!workspace) return fail(SLORR_ERR_WORKSPACE, "workspace is NULL");
    if (reinterpret_cast<uintptr_t>(workspace) % 256 != 0)
        return fail(SLORR_ERR_WORKSPACE, "workspace is not 256-byte aligned");
    if (ws_bytes < h->total_bytes) return fail(SLORR_ERR_WORKSPACE, "workspace too small");
    if (steps < 0 || steps > h->opt.iters) return fail(SLORR_ERR_INVALID_ARG, "steps out of range");
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    s = prepare(h, ws, st);
    if (s != SLORR_OK) return s;
    s = upload_ptrs(h, ws, weights, finish ? grads : nullptr, st);
    if (s != SLORR_OK) return s;
    if ((h->opt.flags & SLORR_FLAG_GRAPH) && finish && !h->timing)
        return launch_graph(h, ws, loss, per, steps, st, descent, eta);
    return launch_all(h, ws, loss, per, steps, finish, st, descent, eta);
}

// Every launch of one call, on `st` (after run() checked the arguments, the
// plan is in the workspace and the pointer arrays are uploaded).
slorr_status launch_all(slorr_handle* h, uint8_t* ws, float* loss, float* per, int steps, bool finish,
                        cudaStream_t st, bool descent, float eta) {
    cudaError_t e = cudaMemsetAsync(ws + h->off_counters, 0, (2 * h->shapes.size() + 1) * 4, st);
    // split-K part counts: each Gram's last parts leave them at zero, but a
    // call that timed out may not have
    if (e == cudaSuccess && h->total_split_parts > 0)
        e = cudaMemsetAsync(ws + h->off_split_cnt, 0, size_t(h->total_split_parts) * 16 * 4, st);
    if (e != cudaSuccess) return cuda_fail(e, "counter reset");

    const bool use_tc = h->opt.compute != SLORR_COMPUTE_FP32 && !(h->opt.flags & SLORR_FLAG_SIMT_GEMM);
    const bool fuse_norm = use_tc && fused_norm(h);
    MemLaunch mp = mem_params(h, ws, loss, per, 0);
    MemLaunch cp = mp;  // tiles of the padded iterate
    cp.items = reinterpret_cast<const MemItem*>(ws + h->off_x_items);
    cp.num_items = int(h->x_items.size());
    if (fuse_norm) {
        cp.tile_base = reinterpret_cast<const int32_t*>(ws + h->off_xtilebase);
        cp.tile_count = reinterpret_cast<const int32_t*>(ws + h->off_xtilecount);
        Traced tr(h, 7, st);
        if ((e = launch_normcast(cp, st)) != cudaSuccess) return cuda_fail(e, "normcast launch");
        if ((e = launch_finalize(cp, 2, st)) != cudaSuccess) return cuda_fail(e, "finalize launch");
        tr.done(2);
    } else {
        mp.items = reinterpret_cast<const MemItem*>(ws + h->off_w_items);
        mp.num_items = int(h->w_items.size());
        {
            Traced tr(h, 0, st);
            if ((e = launch_sumsq(mp, st)) != cudaSuccess) return cuda_fail(e, "sumsq launch");
            if ((e = launch_finalize(mp, 0, st)) != cudaSuccess) return cuda_fail(e, "finalize launch");
            tr.done(2);
        }
        Traced tr(h, 1, st);
        if ((e = launch_cast(cp, st)) != cudaSuccess) return cuda_fail(e, "cast launch");
        if (tf32_tc(h)) {
            // fp32 mode on the tensor cores: X_0 into hi/lo operand pairs, both orientations
            e = launch_tf32_split(reinterpret_cast<const MatDev*>(ws + h->off_mats),
                                  reinterpret_cast<const MatTf32*>(ws + h->off_tf32_mats), int(h->shapes.size()),
                                  h->tf32_split_tiles, st);
            if (e != cudaSuccess) return cuda_fail(e, "split launch");
            tr.done(2);
        } else {
            tr.done();
        }
    }

    GemmLaunch g{};
    g.mats = reinterpret_cast<const MatDev*>(ws + h->off_mats);
    g.maps = ws + h->off_maps;
    g.status = reinterpret_cast<uint32_t*>(ws + h->off_status);
    g.timeout_ns = static_cast<unsigned long long>(h->opt.timeout_s * 1e9);
    g.test_stall = (h->opt.flags & SLORR_FLAG_TEST_STALL) ? 1 : 0;
    g.pdl = use_pdl(h) ? 1 : 0;
    g.fused_norm = fuse_norm ? 1 : 0;
    g.scalars = reinterpret_cast<const MatScalars*>(ws + h->off_scalars);
    g.split_part = reinterpret_cast<float*>(ws + h->off_split_part);
    g.split_cnt = reinterpret_cast<uint32_t*>(ws + h->off_split_cnt);
    g.coef = reinterpret_cast<const float*>(ws + h->off_coef);
    g.tf32 = reinterpret_cast<const MatTf32*>(ws + h->off_tf32_mats);
    g.tf32_maps = ws + h->off_tf32_maps;
    g.split = split16(h) ? 1 : 0;
    g.last_step = h->opt.iters - 1;
    if (use_tc && dataflow(h) && steps > 0) {
        // every phase of every step in one launch, ordered by completion counts
        g.items = reinterpret_cast<const GemmItem*>(ws + h->off_df_items);
        g.num_items = int(h->df_items.size());
        g.step = -1;
        g.steps = steps;
        g.pair_begin = reinterpret_cast<const int32_t*>(ws + h->off_df_pair_begin);
        g.done = reinterpret_cast<uint32_t*>(ws + h->off_done);
        Traced tr(h, 8, st);
        e = launch_gemm_tc_pair(g, h->elem, h->num_sms, st, -1, h->df_pairs);
        if (e != cudaSuccess) return cuda_fail(e, "gemm launch");
        tr.done();
    } else {
        for (int t = 0; t < steps; ++t) {
            g.step = t;
            for (int ph = 0; ph < 3; ++ph) {
                Traced tr(h, 2 + ph, st);
                if (use_tc) {
                    g.items = reinterpret_cast<const GemmItem*>(ws + h->off_tc_items[ph]);
                    g.num_items = int(h->tc_items[ph].size());
                    e = launch_gemm_tc_pair(g, h->elem, h->num_sms, st, ph, 0);
                } else if (tf32_tc(h)) {
                    g.items = reinterpret_cast<const GemmItem*>(ws + h->off_tf32_items[ph]);
                    g.num_items = int(h->tf32_items[ph].size());
                    e = launch_gemm_tf32(g, ph, st);
                } else {
                    g.items = reinterpret_cast<const GemmItem*>(ws + h->off_simt_items[ph]);
                    g.num_items = int(h->simt_items[ph].size());
                    e = launch_gemm_simt(g, h->elem, st);
                }
                if (e != cudaSuccess) return cuda_fail(e, "gemm launch");
                tr.done();
            }
        }
    }
    if (!finish) return SLORR_OK;
    MemLaunch dp = mem_params(h, ws, loss, per, steps & 1);
    if (split16(h) && steps == h->opt.iters) dp.elem = kF16;  // the last Update stored X_T in fp16
    if (descent) {
        dp.out_mode = kOutDescent;
        dp.grad_scale = -eta * h->opt.grad_scale;  // alpha, beta then carry -eta * lambda * grad_scale
    }
    dp.items = reinterpret_cast<const MemItem*>(ws + h->off_w_items);
    dp.num_items = int(h->w_items.size());
    {
        Traced tr(h, 5, st);
        if ((e = launch_dot(dp, st)) != cudaSuccess) return cuda_fail(e, "dot launch");
        if ((e = launch_finalize(dp, 1, st)) != cudaSuccess) return cuda_fail(e, "finalize launch");
        tr.done(2);
    }
    {
        Traced tr(h, 6, st);
        if ((e = launch_combine(dp, st)) != cudaSuccess) return cuda_fail(e, "combine launch");
        tr.done();
    }
    return SLORR_OK;
}

// Reads and clears the device status word of a workspace (after the caller
// synchronised the stream that used it).
slorr_status take_status_word(const slorr_handle* h, const void* workspace, uint32_t* word) {
    uint8_t* ws = static_cast<uint8_t*>(const_cast<void*>(workspace));
    cudaError_t e = cudaMemcpy(word, ws + h->off_status, 4, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = cudaMemset(ws + h->off_status, 0, 4);
    if (e != cudaSuccess) return cuda_fail(e, "status read");
    return SLORR_OK;
}

slorr_status status_from_word(uint32_t word) {
    if (word & kStatusTimeout) return fail(SLORR_ERR_TIMEOUT, "a device-side wait timed out");
    if (word & kStatusNonFinite) return fail(SLORR_ERR_NONFINITE, "non-finite norm or estimate");
    if (word & kStatusInternal)
        return fail(SLORR_ERR_UNSUPPORTED, "the two CTAs of a tensor-core pair received different TMEM addresses");
    return SLORR_OK;
}

}  // namespace

extern "C" {

void slorr_default_options(slorr_options* o) {
    if (!o) return;
    std::memset(o, 0, sizeof(*o));
    o->variant = SLORR_HOYER;
    o->compute = SLORR_COMPUTE_FP16;
    o->dtype = SLORR_F32;
    o->iters = 6;
    o->ell = 1e-3;
    o->cushion = -1.0;
    o->safety = 1.01;
    o->lambda = 1.0f;
    o->eps = 1e-7f;
    o->grad_scale = 1.0f;
    o->flags = 0;
    o->timeout_s = 2.0;
}

slorr_status slorr_create(slorr_handle** out, const slorr_shape* shapes, int32_t count, const slorr_options* opt) {
    if (!out) return fail(SLORR_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!shapes) return fail(SLORR_ERR_INVALID_ARG, "shapes is NULL");
    if (count < 1 || count > kMaxMatrices) return fail(SLORR_ERR_INVALID_ARG, "count must be in [1, 4096]");
    slorr_options o;
    if (opt)
        o = *opt;
    else
        slorr_default_options(&o);
    std::string why;
    if (!valid_options(o, &why)) return fail(SLORR_ERR_INVALID_ARG, "bad option: " + why);
    for (int i = 0; i < count; ++i)
        if (shapes[i].m < 1 || shapes[i].n < 1 || shapes[i].m > 65536 || shapes[i].n > 65536)
            return fail(SLORR_ERR_INVALID_ARG, "matrix dimensions must be in [1, 65536]");
    auto* h = new slorr_handle();
    h->opt = o;
    h->shapes.assign(shapes, shapes + count);
    h->coeffs.resize(size_t(3) * o.iters);
    if (!host::pe_schedule(o.iters, o.ell, o.cushion, o.safety, h->coeffs.data())) {
        delete h;
        return fail(SLORR_ERR_INVALID_ARG, "Polar Express schedule could not be built");
    }
    if (o.compute == SLORR_COMPUTE_FP32) {
        h->elem = kF32;
        h->esize = 4;
    } else {
        h->elem = (o.compute == SLORR_COMPUTE_BF16 || o.compute == SLORR_COMPUTE_BF16_SPLIT) ? kBF16 : kF16;
        h->esize = 2;
    }
    build_plan(h);
    for (const Geom& g : h->geom)
        if (g.tile_count > 65535 || g.xtile_count > 65535) {
            delete h;
            return fail(SLORR_ERR_UNSUPPORTED, "matrix too large: more than 65535 tiles of 16 x 512 elements");
        }
    *out = h;
    return SLORR_OK;
}

slorr_status slorr_executed_flops(const slorr_handle* h, double* out) {
    if (!h || !out) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    const bool tf32 = tf32_tc(h);
    const bool simt = !tf32 && (h->opt.compute == SLORR_COMPUTE_FP32 || (h->opt.flags & SLORR_FLAG_SIMT_GEMM));
    double total = 0.0;
    for (int ph = 0; ph < 3; ++ph) {
        for (const GemmItem& it : tf32 ? h->tf32_items[ph] : simt ? h->simt_items[ph] : h->tc_items[ph]) {
            const Geom& g = h->geom[it.mat];
            const int Kfull = ph == kGram ? g.Qpad : g.Ppad;
            int kb0, kb1;
            split_range(it, Kfull / kPairBK, &kb0, &kb1);
            const double K = it.ksplit ? double(kb1 - kb0) * kPairBK : double(Kfull);
            const double rows = (simt || tf32) ? double(it.msz) : 256.0;  // pair UMMAs are always M = 256
            // three products per product: fp32 mode (tf32) and bf16 hi/lo mode
            const bool three = tf32 || split16(h);
            total += (three ? 3.0 : 1.0) * 2.0 * rows * double(it.nsz) * K;
        }
    }
    *out = total * double(h->opt.iters);
    return SLORR_OK;
}

slorr_status slorr_gemm_items(const slorr_handle* h, int32_t phase, int32_t* items) {
    if (!h || !items) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    if (phase < 0 || phase > 2) return fail(SLORR_ERR_INVALID_ARG, "phase must be 0 (Gram), 1 (Poly) or 2 (Update)");
    const bool simt = h->opt.compute == SLORR_COMPUTE_FP32 || (h->opt.flags & SLORR_FLAG_SIMT_GEMM);
    *items = int32_t(tf32_tc(h) ? h->tf32_items[phase].size()
                                : simt ? h->simt_items[phase].size() : h->tc_items[phase].size());
    return SLORR_OK;
}

slorr_status slorr_gemm_item_list(const slorr_handle* h, int32_t phase, int32_t* out, int32_t capacity) {
    if (!h || !out) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    if (phase < 0 || phase > 2) return fail(SLORR_ERR_INVALID_ARG, "phase must be 0 (Gram), 1 (Poly) or 2 (Update)");
    const bool simt = h->opt.compute == SLORR_COMPUTE_FP32 || (h->opt.flags & SLORR_FLAG_SIMT_GEMM);
    const std::vector<GemmItem>& v =
        tf32_tc(h) ? h->tf32_items[phase] : simt ? h->simt_items[phase] : h->tc_items[phase];
    if (capacity < int64_t(v.size()) * 7) return fail(SLORR_ERR_INVALID_ARG, "capacity too small");
    for (size_t i = 0; i < v.size(); ++i) {
        const GemmItem& it = v[i];
        const int parts = it.ksplit >> 8;
        int32_t* o = out + i * 7;
        o[0] = it.mat;
        o[1] = it.tm;
        o[2] = it.tn;
        o[3] = it.msz;
        o[4] = it.nsz;
        o[5] = parts > 1 ? (it.ksplit & 0xff) : 0;
        o[6] = parts > 1 ? parts : 1;
    }
    return SLORR_OK;
}

slorr_status slorr_dataflow_items(const slorr_handle* h, int32_t* out, int32_t capacity, int32_t* npairs,
                                  int32_t* count, double* makespan_k) {
    if (!h || !npairs || !count) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    if (!dataflow(h)) return fail(SLORR_ERR_INVALID_ARG, "this handle runs per-phase launches");
    *npairs = h->df_pairs;
    *count = int32_t(h->df_items.size());
    if (makespan_k) *makespan_k = h->df_makespan;
    if (!out) return SLORR_OK;
    if (int64_t(capacity) < int64_t(h->df_items.size()) * 10) return fail(SLORR_ERR_INVALID_ARG, "capacity too small");
    for (int q = 0; q < h->df_pairs; ++q)
        for (int32_t i = h->df_pair_begin[size_t(q)]; i < h->df_pair_begin[size_t(q) + 1]; ++i) {
            const GemmItem& it = h->df_items[size_t(i)];
            const int parts = it.ksplit >> 8;
            int32_t* o = out + size_t(i) * 10;
            o[0] = q;
            o[1] = h->df_seq[size_t(i)];
            o[2] = it.step;
            o[3] = it.phase;
            o[4] = it.mat;
            o[5] = it.tm;
            o[6] = it.tn;
            o[7] = parts > 1 ? (it.ksplit & 0xff) : 0;
            o[8] = parts > 1 ? parts : 1;
            o[9] = int32_t(it.wait);
        }
    return SLORR_OK;
}

slorr_status slorr_gemm_pair_load(const slorr_handle* h, int32_t phase, int32_t npairs, int64_t* max_k,
                                  int64_t* total_k) {
    if (!h || !max_k || !total_k) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    if (phase < 0 || phase > 2) return fail(SLORR_ERR_INVALID_ARG, "phase must be 0 (Gram), 1 (Poly) or 2 (Update)");
    if (npairs < 1) return fail(SLORR_ERR_INVALID_ARG, "npairs must be >= 1");
    std::vector<int64_t> load(size_t(npairs), 0);
    const std::vector<GemmItem>& v = h->tc_items[phase];
    for (size_t i = 0; i < v.size(); ++i) {
        const Geom& g = h->geom[v[i].mat];
        const int K = phase == kGram ? g.Qpad : g.Ppad;
        int b, e;
        split_range(v[i], K / kPairBK, &b, &e);
        load[i % size_t(npairs)] += int64_t(e - b) * kPairBK;
    }
    *max_k = *std::max_element(load.begin(), load.end());
    *total_k = std::accumulate(load.begin(), load.end(), int64_t(0));
    return SLORR_OK;
}

slorr_status slorr_workspace_size(const slorr_handle* h, size_t* bytes) {
    if (!h || !bytes) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    *bytes = h->total_bytes;
    return SLORR_OK;
}

slorr_status slorr_reg_forward_backward(slorr_handle* h, const void* const* weights, void* const* grads,
                                        float* loss_out, float* per_matrix_out, void* workspace,
                                        size_t workspace_bytes, void* stream) {
    if (!h) return fail(SLORR_ERR_INVALID_ARG, "handle is NULL");
    return run(h, weights, grads, loss_out, per_matrix_out, workspace, workspace_bytes, h->opt.iters, true,
               static_cast<cudaStream_t>(stream));
}

slorr_status slorr_reg_descent_step(slorr_handle* h, void* const* weights, float eta, float* loss_out,
                                    float* per_matrix_out, void* workspace, size_t workspace_bytes,
                                    void* stream) {
    if (!h) return fail(SLORR_ERR_INVALID_ARG, "handle is NULL");
    return run(h, const_cast<const void* const*>(weights), nullptr, loss_out, per_matrix_out, workspace,
               workspace_bytes, h->opt.iters, true, static_cast<cudaStream_t>(stream), true, eta);
}

slorr_status slorr_reset_workspace(slorr_handle* h) {
    if (!h) return fail(SLORR_ERR_INVALID_ARG, "handle is NULL");
    h->prepared_ws = nullptr;
    h->last_ptrs.clear();
    return SLORR_OK;
}

slorr_status slorr_get_status(slorr_handle* h, const void* workspace, void* stream) {
    if (!h || !workspace) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    uint32_t word = 0;
    slorr_status s = take_status_word(h, workspace, &word);
    if (s != SLORR_OK) return s;
    return status_from_word(word);
}

slorr_status slorr_run_steps(slorr_handle* h, const void* const* weights, void* workspace, size_t workspace_bytes,
                             int32_t steps, void* stream) {
    return run(h, weights, nullptr, nullptr, nullptr, workspace, workspace_bytes, steps, false,
               static_cast<cudaStream_t>(stream));
}

slorr_status slorr_iterate_view(const slorr_handle* h, const void* workspace, int32_t i, int32_t after_steps,
                                slorr_matrix_view* out) {
    if (!h || !workspace || !out) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    if (i < 0 || i >= int(h->shapes.size())) return fail(SLORR_ERR_INVALID_ARG, "matrix index out of range");
    if (after_steps < 0 || after_steps > h->opt.iters) return fail(SLORR_ERR_INVALID_ARG, "steps out of range");
    const Geom& g = h->geom[i];
    const uint8_t* ws = static_cast<const uint8_t*>(workspace);
    out->x = ws + g.off_x[after_steps & 1];
    out->rows = g.m;
    out->cols = g.n;
    out->ld = g.ld;
    // bf16 hi/lo mode: the high parts, and X_T (after the last step) in fp16
    out->elem = (split16(h) && after_steps == h->opt.iters) ? kF16 : h->elem;
    out->transposed = g.transposed;
    const MatScalars* sc = reinterpret_cast<const MatScalars*>(ws + h->off_scalars) + i;
    out->frob_sq = &sc->frob_sq;
    out->n_hat = &sc->n_hat;
    out->x0_scale = &sc->x0_scale;
    return SLORR_OK;
}

slorr_status slorr_get_coefficients(const slorr_handle* h, double* abc, int32_t capacity) {
    if (!h || !abc) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    if (capacity < int(h->coeffs.size())) return fail(SLORR_ERR_INVALID_ARG, "capacity too small");
    std::copy(h->coeffs.begin(), h->coeffs.end(), abc);
    return SLORR_OK;
}

slorr_status slorr_pe_coefficients(int32_t iters, double ell, double cushion, double safety, double* abc) {
    if (!abc) return fail(SLORR_ERR_INVALID_ARG, "abc is NULL");
    if (iters < 1 || iters > kMaxIters) return fail(SLORR_ERR_INVALID_ARG, "iters must be in [1, 16]");
    if (!host::pe_schedule(iters, ell, cushion, safety, abc))
        return fail(SLORR_ERR_INVALID_ARG, "Polar Express schedule could not be built");
    return SLORR_OK;
}

double slorr_cushion_ratio(void) { return host::cushion_ratio(); }

int64_t slorr_flops(const slorr_shape* shapes, int32_t count, int32_t iters) {
    if (!shapes || count < 0 || iters < 0) return -1;
    int64_t total = 0;
    for (int i = 0; i < count; ++i) {
        const int64_t P = std::min(shapes[i].m, shapes[i].n), Q = std::max(shapes[i].m, shapes[i].n);
        total += 4 * P * P * Q + 2 * P * P * P;
    }
    return total * iters;
}

slorr_status slorr_partition(const slorr_shape* shapes, int32_t count, int32_t world, int32_t rank,
                             int32_t* out_indices, int32_t* out_count) {
    if (!shapes || !out_indices || !out_count || count < 0) return fail(SLORR_ERR_INVALID_ARG, "bad argument");
    if (world < 1 || rank < 0 || rank >= world) return fail(SLORR_ERR_INVALID_ARG, "bad world/rank");
    std::vector<int> order(count);
    std::iota(order.begin(), order.end(), 0);
    auto cost = [&](int i) { return slorr_flops(&shapes[i], 1, 1); };
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost(a) > cost(b); });
    std::vector<int64_t> load(world, 0);
    std::vector<int> owner(count, 0);
    for (int i : order) {
        int best = 0;
        for (int r = 1; r < world; ++r)
            if (load[r] < load[best]) best = r;
        owner[i] = best;
        load[best] += cost(i);
    }
    int k = 0;
    for (int i = 0; i < count; ++i)
        if (owner[i] == rank) out_indices[k++] = i;
    *out_count = k;
    return SLORR_OK;
}

slorr_status slorr_set_timing(slorr_handle* h, int32_t enable) {
    if (!h) return fail(SLORR_ERR_INVALID_ARG, "handle is NULL");
    h->timing = enable != 0;
    return SLORR_OK;
}

slorr_status slorr_read_timing(slorr_handle* h, double* ms, int64_t* launches, int32_t kinds) {
    if (!h || !ms || !launches || kinds < 1 || kinds > SLORR_NUM_KERNEL_KINDS)
        return fail(SLORR_ERR_INVALID_ARG, "bad argument");
    slorr_status s = SLORR_OK;
    for (auto& m : h->marks) {
        float t = 0.f;
        cudaError_t e = cudaEventSynchronize(m.stop);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&t, m.start, m.stop);
        if (e != cudaSuccess && s == SLORR_OK) s = cuda_fail(e, "event timing");
        if (m.kind < kinds) {
            ms[m.kind] += double(t);
            launches[m.kind] += m.kernels;
        }
        h->ev_pool.push_back(m.start);
        h->ev_pool.push_back(m.stop);
    }
    h->marks.clear();
    return s;
}

void slorr_destroy(slorr_handle* h) { delete h; }

const char* slorr_status_string(slorr_status s) {
    switch (s) {
        case SLORR_OK: return "ok";
        case SLORR_ERR_INVALID_ARG: return "invalid argument";
        case SLORR_ERR_UNSUPPORTED: return "unsupported";
        case SLORR_ERR_CUDA: return "CUDA error";
        case SLORR_ERR_WORKSPACE: return "workspace missing or too small";
        case SLORR_ERR_TIMEOUT: return "device wait timed out";
        case SLORR_ERR_NONFINITE: return "non-finite value";
    }
    return "unknown status";
}

const char* slorr_last_error(void) { return g_last_error.c_str(); }

}  // extern "C"

// ---- host-resident weight sets: the copy / compute pipeline ----------------------

struct slorr_pipeline {
    std::vector<slorr_handle*> groups;  // one plan per run of consecutive matrices
    std::vector<int> first;             // first matrix of each group; first[G] = count
    std::vector<size_t> ws_off;         // offset of each group's workspace slice
    std::vector<size_t> bytes;          // bytes of W_i (and of its grad)
    size_t off_loss = 0;                // G partial losses, the total, `count` per-matrix values
    size_t total_bytes = 0;
    int count = 0;
    int device = -1;                    // streams and events live on this device
    cudaStream_t s_in = nullptr, s_out = nullptr;
    cudaEvent_t ev_start = nullptr, ev_out = nullptr;
    std::vector<cudaEvent_t> ev_in, ev_done;
    ~slorr_pipeline() {
        for (auto* g : groups) delete g;
        for (auto e : ev_in) cudaEventDestroy(e);
        for (auto e : ev_done) cudaEventDestroy(e);
        if (ev_start) cudaEventDestroy(ev_start);
        if (ev_out) cudaEventDestroy(ev_out);
        if (s_in) cudaStreamDestroy(s_in);
        if (s_out) cudaStreamDestroy(s_out);
    }
};

namespace {

// Streams and events, created on the current device at the first run.
slorr_status pipeline_init(slorr_pipeline* p) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (p->device >= 0) {
        if (dev != p->device) return fail(SLORR_ERR_INVALID_ARG, "pipeline used on another device than its first run");
        return SLORR_OK;
    }
    const int G = int(p->groups.size());
    e = cudaStreamCreateWithFlags(&p->s_in, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p->s_out, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->ev_start, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->ev_out, cudaEventDisableTiming);
    for (int g = 0; g < G && e == cudaSuccess; ++g) {
        cudaEvent_t a = nullptr, b = nullptr;
        e = cudaEventCreateWithFlags(&a, cudaEventDisableTiming);
        if (e == cudaSuccess) {
            p->ev_in.push_back(a);
            e = cudaEventCreateWithFlags(&b, cudaEventDisableTiming);
            if (e == cudaSuccess) p->ev_done.push_back(b);
        }
    }
    if (e != cudaSuccess) return cuda_fail(e, "pipeline stream / event creation");
    p->device = dev;
    return SLORR_OK;
}

}  // namespace

extern "C" {

slorr_status slorr_pipeline_create(slorr_pipeline** out, const slorr_shape* shapes, int32_t count,
                                   const slorr_options* opt, int32_t groups) {
    if (!out) return fail(SLORR_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (groups < 1) return fail(SLORR_ERR_INVALID_ARG, "groups must be >= 1");
    // validates shapes, count and options
    slorr_handle* probe = nullptr;
    slorr_status s = slorr_create(&probe, shapes, count, opt);
    if (s != SLORR_OK) return s;
    const int esz = probe->opt.dtype == SLORR_BF16 ? 2 : 4;
    delete probe;
    auto* p = new slorr_pipeline();
    p->count = count;
    size_t total = 0;
    for (int i = 0; i < count; ++i) {
        p->bytes.push_back(size_t(shapes[i].m) * size_t(shapes[i].n) * size_t(esz));
        total += p->bytes.back();
    }
    // Consecutive runs of about total / G bytes each, none empty.
    const int G = std::min<int>(groups, count);
    p->first.push_back(0);
    size_t acc = 0;
    for (int i = 0; i < count; ++i) {
        acc += p->bytes[i];
        const int g = int(p->first.size());  // group being filled is g - 1
        const int left = count - (i + 1);     // matrices not yet assigned
        const int needed = G - g;             // groups still to start after this one
        if (g < G && (acc * size_t(G) >= total * size_t(g) || left == needed) && left >= needed)
            p->first.push_back(i + 1);
    }
    p->first.push_back(count);
    size_t off = 0;
    for (size_t g = 0; g + 1 < p->first.size(); ++g) {
        slorr_handle* h = nullptr;
        s = slorr_create(&h, shapes + p->first[g], p->first[g + 1] - p->first[g], opt);
        if (s != SLORR_OK) {
            delete p;
            return s;
        }
        p->groups.push_back(h);
        p->ws_off.push_back(off);
        off = align_up(off + h->total_bytes, 1024);
    }
    p->off_loss = off;
    off = align_up(off + (p->groups.size() + 1 + size_t(count)) * sizeof(float), 256);
    p->total_bytes = off;
    *out = p;
    return SLORR_OK;
}

slorr_status slorr_pipeline_workspace_size(const slorr_pipeline* p, size_t* bytes) {
    if (!p || !bytes) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    *bytes = p->total_bytes;
    return SLORR_OK;
}

slorr_status slorr_pipeline_forward_backward(slorr_pipeline* p, const void* const* host_weights,
                                             void* const* host_grads, float* host_loss, float* host_per_matrix,
                                             void* const* dev_weights, void* const* dev_grads, void* workspace,
                                             size_t workspace_bytes, void* stream) {
    if (!p) return fail(SLORR_ERR_INVALID_ARG, "pipeline is NULL");
    if (!host_weights || !host_grads || !host_loss || !dev_weights || !dev_grads)
        return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    for (int i = 0; i < p->count; ++i)
        if (!host_weights[i] || !host_grads[i]) return fail(SLORR_ERR_INVALID_ARG, "host pointer is NULL");
    if (!workspace) return fail(SLORR_ERR_WORKSPACE, "workspace is NULL");
    if (reinterpret_cast<uintptr_t>(workspace) % 256 != 0)
        return fail(SLORR_ERR_WORKSPACE, "workspace is not 256-byte aligned");
    if (workspace_bytes < p->total_bytes) return fail(SLORR_ERR_WORKSPACE, "workspace too small");
    slorr_status s = pipeline_init(p);
    if (s != SLORR_OK) return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    float* parts = reinterpret_cast<float*>(ws + p->off_loss);
    const int G = int(p->groups.size());
    float* total = parts + G;
    float* per = total + 1;
    // Copies start after the caller's earlier work on `stream`.
    cudaError_t e = cudaEventRecord(p->ev_start, st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_in, p->ev_start, 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(p->s_out, p->ev_start, 0);
    // in: every group's weights and grads, in group order
    for (int g = 0; g < G && e == cudaSuccess; ++g) {
        for (int i = p->first[g]; i < p->first[g + 1] && e == cudaSuccess; ++i) {
            e = cudaMemcpyAsync(dev_weights[i], host_weights[i], p->bytes[i], cudaMemcpyHostToDevice, p->s_in);
            if (e == cudaSuccess)
                e = cudaMemcpyAsync(dev_grads[i], host_grads[i], p->bytes[i], cudaMemcpyHostToDevice, p->s_in);
        }
        if (e == cudaSuccess) e = cudaEventRecord(p->ev_in[g], p->s_in);
    }
    if (e != cudaSuccess) return cuda_fail(e, "pipeline copy-in");
    // compute: group g once its copies have landed
    for (int g = 0; g < G; ++g) {
        e = cudaStreamWaitEvent(st, p->ev_in[g], 0);
        if (e != cudaSuccess) return cuda_fail(e, "pipeline wait");
        slorr_handle* h = p->groups[g];
        const int f = p->first[g];
        s = run(h, reinterpret_cast<const void* const*>(dev_weights + f), dev_grads + f, parts + g, per + f,
                ws + p->ws_off[g], h->total_bytes, h->opt.iters, true, st);
        if (s != SLORR_OK) return s;
        e = cudaEventRecord(p->ev_done[g], st);
        if (e != cudaSuccess) return cuda_fail(e, "pipeline record");
    }
    // out: each group's grads once its kernels are done
    for (int g = 0; g < G && e == cudaSuccess; ++g) {
        e = cudaStreamWaitEvent(p->s_out, p->ev_done[g], 0);
        for (int i = p->first[g]; i < p->first[g + 1] && e == cudaSuccess; ++i)
            e = cudaMemcpyAsync(host_grads[i], dev_grads[i], p->bytes[i], cudaMemcpyDeviceToHost, p->s_out);
    }
    if (e == cudaSuccess) e = cudaEventRecord(p->ev_out, p->s_out);
    if (e != cudaSuccess) return cuda_fail(e, "pipeline copy-out");
    // the loss (partial losses added in group order) and the per-matrix values
    e = launch_sum_parts(parts, G, total, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(host_loss, total, sizeof(float), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && host_per_matrix)
        e = cudaMemcpyAsync(host_per_matrix, per, size_t(p->count) * sizeof(float), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, p->ev_out, 0);
    if (e != cudaSuccess) return cuda_fail(e, "pipeline finish");
    return SLORR_OK;
}

slorr_status slorr_pipeline_get_status(slorr_pipeline* p, const void* workspace, void* stream) {
    if (!p || !workspace) return fail(SLORR_ERR_INVALID_ARG, "NULL argument");
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    uint32_t all = 0;
    for (size_t g = 0; g < p->groups.size(); ++g) {
        uint32_t word = 0;
        slorr_status s = take_status_word(p->groups[g], static_cast<const uint8_t*>(workspace) + p->ws_off[g], &word);
        if (s != SLORR_OK) return s;
        all |= word;
    }
    return status_from_word(all);
}

void slorr_pipeline_destroy(slorr_pipeline* p) { delete p; }

}  // extern "C"
