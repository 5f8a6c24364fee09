// Internal declarations shared by libslorr's translation units.
//
// Device-side plan: for each weight matrix W_i (m x n) the Polar Express
// iterate X is P x Q with P = min(m, n), Q = max(m, n) (Sec. 3 "Computational
// cost": the Gram matrix is formed on the min side).  It is stored in W's own
// orientation -- row-major [m][n], i.e. as X^T when m > n -- so that the norm,
// cast, dot and gradient passes are elementwise; the tensor-core kernel reads
// it as a K-major or MN-major operand as each phase needs.  Both dimensions
// are zero-padded: P to Ppad and Q to Qpad (multiples of 128).  Zero padding is exact: zero rows/columns of X give zero rows/columns
// of A = X X^T; M = a I + b A + c A^2 is a I on the padded block, which only
// ever multiplies zero rows of X; and the odd polynomial maps zero to zero
// (App. B, "zero singular values stay zero").
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>
#include <utility>

#include <cuda_runtime.h>

namespace slorr {

constexpr int kMaxMatrices = 4096;
constexpr int kMaxIters = 16;
constexpr int kPadRows = 128;   // Ppad granularity (tcgen05 tile M)
constexpr int kPadCols = 128;   // Qpad granularity (a CTA pair splits a tile's 2 x 64 columns)
// K block of one stage of the CTA-pair GEMM: two 128-byte swizzle atoms of
// 16-bit elements (Ppad and Qpad are multiples of it)
constexpr int kPairBK = 128;

// Element type of the iterate buffers X, A, B.
enum Elem : int32_t { kF32 = 0, kF16 = 1, kBF16 = 2 };

// Status bits written by kernels into the workspace status word.
// kStatusInternal: the two CTAs of a pair received different TMEM addresses
// (the pair kernel then does no work).
enum StatusBits : uint32_t { kStatusTimeout = 1u, kStatusNonFinite = 2u, kStatusInternal = 4u };

// Per-matrix device descriptor (lives in the workspace).
struct MatDev {
    void* x[2];        // ping-pong iterate buffers, rows x ld in W's orientation
    void* a;           // A = X X^T, Ppad x Ppad
    void* b;           // M = a I + b A + c A^2, Ppad x Ppad
    // bf16 hi/lo mode (SLORR_COMPUTE_BF16_SPLIT): x[], a and b hold bf16(v)
    // and these the residuals bf16(v - bf16(v)) of the iterates, of A and of M
    // (null in the other modes)
    void* xlo[2];
    void* alo;
    void* blo;
    int32_t m, n;      // shape of W
    int32_t P, Q;      // min / max
    int32_t Ppad, Qpad;
    int32_t transposed;  // 1 when m > n: the buffer holds X^T (Qpad x Ppad)
    int32_t rows;      // buffer rows: Ppad, or Qpad when transposed
    int32_t ld;        // buffer row length: Qpad, or Ppad when transposed
    int32_t pad_;
};

// fp32 mode on the tensor cores (three-pass TF32): every product operand is
// kept as a pair (hi, lo) of fp32 arrays holding tf32 values, hi = tf32(v) and
// lo = tf32(v - hi), both rounded to nearest.  All operands are K-major: the
// iterate is kept both in the Gram orientation (P x Q, for the Gram product)
// and transposed (Q x P, the B operand of the update M X).
struct MatTf32 {
    void* xg[2][2];    // [buffer][hi, lo]: X, Ppad x Qpad row-major
    void* xu[2][2];    // [buffer][hi, lo]: X^T, Qpad x Ppad row-major
    void* a[2];        // [hi, lo]: A, Ppad x Ppad
    void* m[2];        // [hi, lo]: M, Ppad x Ppad
};
// Tensor maps per matrix of the fp32 tensor-core path (32 x 64-element boxes):
// xg[b][h] at 2 b + h, xu[b][h] at 4 + 2 b + h, a[h] at 8 + h, m[h] at 10 + h.
constexpr int kTf32MapsPerMatrix = 12;

// Per-matrix scalars (workspace).
struct MatScalars {
    double frob_sq;    // ||W||_F^2
    double n_hat;      // sum(W * P_hat)
    float scale;       // 1 / (||W||_F + eps): the normalisation of X_0
    float x0_scale;    // X_0 = x0_scale * (the stored X_0 buffer): scale when the
                       // fused norm pass stored W unscaled, else 1
    float alpha;       // gradient = alpha * P_hat - beta * W (lambda, grad_scale included)
    float beta;
    int32_t skip;      // non-finite norm or estimate: leave the gradient untouched
    int32_t pad_;
};

// One output tile of a grouped GEMM phase.
struct GemmItem {
    uint16_t mat;
    uint16_t tm;       // row tile index (256 rows per tcgen05 tile, 32 for SIMT)
    uint16_t tn;       // column tile index (256 columns per tcgen05 tile, 32 for SIMT)
    uint16_t nsz;      // columns in this tile
    uint16_t msz;      // rows in this tile
    uint16_t ksplit;   // split K (CTA-pair Gram): part s | (parts S << 8); 0 = whole K
    uint32_t sid;      // split K: the tile's first 256 x 256 partial slot (parts sid .. sid + S - 1)
    uint8_t step;      // Polar Express step t of this item (dataflow launch; 0 in per-phase lists)
    uint8_t phase;     // kGram, kPoly or kUpdate
    uint16_t pad_;
    uint32_t wait;     // dataflow launch: the item may start once done[mat] >= wait
};

// K blocks [begin, end) of an item's nkb: part s of S takes an equal share.
__host__ __device__ inline void split_range(const GemmItem& it, int nkb, int* begin, int* end) {
    const int parts = it.ksplit >> 8;
    if (parts <= 1) {
        *begin = 0;
        *end = nkb;
        return;
    }
    const int s = it.ksplit & 0xff;
    *begin = s * nkb / parts;
    *end = (s + 1) * nkb / parts;
}

#ifndef SLORR_MAX_SPLIT
#define SLORR_MAX_SPLIT 2
#endif
constexpr int kMaxSplit = SLORR_MAX_SPLIT;  // K parts of a split Gram tile (a build-time tuning knob)
constexpr int kSimtTile = 32;              // output tile of the CUDA-core GEMM (32 x 32)

// One chunk of a memory-bound pass: a kMemRows x kMemCols tile of W (or of
// the padded iterate buffer for the cast).
constexpr int kMemRows = 16;
constexpr int kMemCols = 512;
constexpr int kMemVec = 8;      // consecutive columns per thread
struct MemItem {
    uint16_t mat;
    uint16_t tile_r;   // tile row index (kMemRows rows), or kFlatTile
    uint16_t tile_c;   // tile column index (kMemCols cols)
    uint16_t seq;      // index of this tile within its matrix
};
// tile_r of a flat tile: elements [8192 seq, 8192 seq + 8192) of a matrix
// whose rows are a multiple of 128 elements (ld == n), W and the iterate
// buffer at the same offset.
constexpr uint16_t kFlatTile = 0xffff;

// Phases of one Polar Express step (the step's polynomial is applied as
// X <- M X with M = a I + b A + c A^2, the same product as a X + (b A + c A^2) X).
enum Phase : int32_t { kGram = 0, kPoly = 1, kUpdate = 2 };

// Dataflow launch (the default): every Gram, Poly and Update tile of every
// step in one launch.  CTA pair q runs items [pair_begin[q], pair_begin[q + 1])
// in order; each epilogue warp of both CTAs adds 1 to done[mat] once its part
// of an item is stored, and an item's TMA producer waits until done[mat]
// reaches the item's `wait`: the count after every earlier (step, phase) of
// its matrix.  Per-phase launches (pair_begin == nullptr) hand item i to pair
// i mod npairs and run the single step `step`.
constexpr int kDataflowEpiWarps = 8;   // epilogue warps per CTA of the dataflow kernel
constexpr int kDoneIncPerItem = 2 * kDataflowEpiWarps;
constexpr int kMaxPlanPairs = 512;

struct GemmLaunch {
    const GemmItem* items;
    int32_t num_items;
    int32_t step;              // per-phase launch: the step t; dataflow: -1 (each item's own)
    int32_t steps;             // dataflow: items of steps >= steps are skipped
    const float* coef;         // (a_t, b_t, c_t) for t = 0 .. T - 1, 3 T floats (workspace)
    const int32_t* pair_begin; // dataflow: each pair's range of items (npairs + 1 offsets)
    uint32_t* done;            // dataflow: per-matrix completion counts (zeroed before the launch)
    const MatDev* mats;
    const void* maps;          // CUtensorMap array, kMapsPerMatrix per matrix
    uint32_t* status;
    unsigned long long timeout_ns;
    int32_t test_stall;        // 1: the MMA thread first waits on a barrier nothing arrives on
    int32_t pdl;               // launch with programmatic dependent launch
    // fused_norm = 1 (16-bit iterates after the fused norm pass, which stores
    // X_0 as W rounded to 16 bits): in step 0 the Gram epilogue multiplies by
    // scalars[i].x0_scale^2 and the Update epilogue by scalars[i].x0_scale.
    int32_t fused_norm;
    const MatScalars* scalars;
    // split K (CTA-pair Gram): part s of a split tile leaves its fp32 partial
    // at split_part + ((sid + s) * 256 + column) * 256 + row (tile
    // coordinates), and counts it in split_cnt[sid * 16 + rank * 8 + group * 4
    // + quad]; the epilogue warp that counts last adds the parts and stores
    // the tile.
    float* split_part;
    uint32_t* split_cnt;
    // fp32 mode on the tensor cores: the hi/lo operand arrays and their maps
    const MatTf32* tf32;
    const void* tf32_maps;
    // bf16 hi/lo mode: every product takes three bf16 products of the hi/lo
    // parts of its operands (hi hi + lo hi + hi lo), the Gram and the Poly
    // store A and M as hi and lo parts, and the Update stores X' so too,
    // except in step last_step, which stores X_T in fp16 for the dot and
    // combine passes
    int32_t split;
    int32_t last_step;
};

// Tensor maps per matrix: X0, X1, A, M, and in bf16 hi/lo mode the low
// parts X0_lo, X1_lo, M_lo, A_lo (each read as K-major or MN-major halves
// through the same 3-D map).
constexpr int kMapsPerMatrix = 8;

// Where the combine pass puts lambda * grad_scale * G_i.
enum OutMode : int32_t {
    kOutAccumulate = 0,  // grads[i] += (Listing 1 backward, Alg. 2)
    kOutOverwrite = 1,   // grads[i] =  (the pre-update gradient of Alg. 1)
    kOutDescent = 2,     // weights[i] += (grad_scale already holds -eta * grad_scale), in place
};

struct MemLaunch {
    const MemItem* items;
    int32_t num_items;
    const MatDev* mats;
    MatScalars* scalars;
    float* partials;           // one float per (matrix, tile)
    float* partials_max;       // fused norm pass: max |w| per tile
    const int32_t* tile_base;  // first partial index of each matrix
    const int32_t* tile_count; // tiles per matrix
    uint32_t* counters;        // per-matrix completion counters
    uint32_t* status;
    int32_t count;             // matrices
    int32_t cur;               // iterate buffer holding X_0 (cast) or X_T (dot/combine)
    int32_t elem;              // Elem of the iterate
    int32_t wdtype;            // 0 fp32, 1 bf16 weights/grads
    int32_t variant;           // 0 Hoyer, 1 Nuc
    int32_t out_mode;          // kOutAccumulate, kOutOverwrite or kOutDescent
    int32_t pdl;               // launch with programmatic dependent launch
    float eps, lambda, grad_scale;
    float* loss_out;
    float* per_matrix_out;
    const void* const* weights;  // device array of weight pointers
    void* const* grads;          // device array of grad pointers
};

// Launchers (return cudaGetLastError() of the launch).
cudaError_t launch_sumsq(const MemLaunch& p, cudaStream_t s);
cudaError_t launch_cast(const MemLaunch& p, cudaStream_t s);
cudaError_t launch_normcast(const MemLaunch& p, cudaStream_t s);
cudaError_t launch_dot(const MemLaunch& p, cudaStream_t s);
// which: 0 after sumsq, 1 after dot (and the loss), 2 after normcast
cudaError_t launch_finalize(const MemLaunch& p, int which, cudaStream_t s);
cudaError_t launch_combine(const MemLaunch& p, cudaStream_t s);
cudaError_t launch_sum_parts(const float* parts, int n, float* out, cudaStream_t s);
cudaError_t launch_gemm_simt(const GemmLaunch& p, int elem, cudaStream_t s);
// One per-phase launch (phase = kGram, kPoly or kUpdate; npairs ignored) or
// the dataflow launch (phase = -1) over `npairs` CTA pairs.  Gram and Update
// take 4 epilogue warps per CTA, Poly and the dataflow launch, which mixes
// phases, 8.
cudaError_t launch_gemm_tc_pair(const GemmLaunch& p, int elem, int num_sms, cudaStream_t s, int phase,
                                int npairs);
// fp32 mode on the tensor cores: one phase of one step (p.step), one CTA per
// 128 x 64 output tile (kernels_tf32.cu).
cudaError_t launch_gemm_tf32(const GemmLaunch& p, int phase, cudaStream_t s);
// fp32 mode on the tensor cores: splits X_0 (the fp32 iterate buffer x[0], in
// W's orientation) into the hi/lo arrays of both orientations.
cudaError_t launch_tf32_split(const MatDev* mats, const MatTf32* tf32, int count, int max_tiles, cudaStream_t s);
// CTA pairs of the dataflow kernel that can be resident at once on the
// current device (0 and an error when the query fails).
cudaError_t tc_pair_dataflow_capacity(int elem, int num_sms, int* pairs);

#if defined(__CUDACC__)
// Launches `kernel` on `st`; with pdl, as a programmatic dependent of the
// stream's previous kernel (the kernel must call griddep_wait() before it
// reads anything an earlier kernel wrote).
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), unsigned grid, unsigned block, size_t smem, cudaStream_t st,
                          bool pdl, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = pdl ? attr : nullptr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
#endif

// Records the message slorr_last_error() returns on this thread (api.cu).
void set_last_error(const std::string& msg);

// Host Polar Express schedule (schedule.cpp).
namespace host {
bool minimax_quintic(double lo, double hi, double out[4]);
double cushion_ratio();
bool pe_schedule(int T, double ell, double cushion, double safety, double* abc);
}  // namespace host

}  // namespace slorr
