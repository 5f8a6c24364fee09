// Memory-bound passes of the SLORR hot path, grouped over all weight matrices:
//   sumsq   ||W_i||_F^2                                  (Listing 1, frob)
//   cast    X_0 = W_i / (||W_i||_F + eps), zero padded    (Sec. 3 "Computing the polar factor")
//   normcast  sumsq and cast in one read of W, for 16-bit iterates: the
//           buffer receives W itself rounded to 16 bits, and the first Gram
//           and Update epilogues apply the scale (x0_scale); the finalize
//           kernel re-casts, with the scale, a matrix whose values would lose
//           precision in an unscaled fp16 copy
//   dot     n_hat_i = sum(W_i * P_hat_i), values L_i and the loss
//                                                        (Sec. 3 "Computing the nuclear ...", Listing 1)
//   combine W_i.grad += lambda * grad_scale * G_i       (Listing 1 backward, Alg. 2)
//           or, in overwrite mode, out_i = lambda * grad_scale * G_i, the
//           pre-update gradient Alg. 1 (decoupled SLORR) applies after the
//           optimizer step, or, in descent mode, W_i -= eta * lambda *
//           grad_scale * G_i in place (the last line of Alg. 1 with no task
//           update in between: the regularizer-only step of Props. 2 and 3)
// The iterates are stored in W's orientation (row-major, row length `ld`), so
// every pass is elementwise.  A block handles one kMemRows x kMemCols tile:
// each of its 256 threads owns 8 consecutive columns of 4 rows and issues all
// its 128-bit loads before using them.  Rows whose length is not a multiple
// of 8 take a scalar path.  A matrix whose rows are a multiple of 128
// elements has an iterate buffer without column padding (ld == n); its tiles
// are runs of 8192 consecutive elements instead ("flat"), so rows that are
// not a multiple of 512 long leave no thread idle.  Per-matrix coefficients (the cast scale, the
// gradient's alpha and beta) are computed once by the finalize kernels, in
// double precision, and read as floats by the streaming passes.  Cross-tile sums are
// deterministic: each streaming block writes one partial per tile and exits;
// a finalize kernel (one block per matrix) adds a matrix's partials in index
// order in double precision.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"

namespace slorr {
namespace {

constexpr int kThreads = 256;
constexpr int kVecPerRow = kMemCols / kMemVec;       // 64 threads per tile row
constexpr int kRowsPerPass = kThreads / kVecPerRow;  // 4
constexpr int kPasses = kMemRows / kRowsPerPass;     // 4

struct F8 {
    float4 lo, hi;
};

__device__ __forceinline__ float bf2f(uint32_t u16) { return __uint_as_float(u16 << 16); }

__device__ __forceinline__ F8 zero8() {
    F8 z;
    z.lo = make_float4(0.f, 0.f, 0.f, 0.f);
    z.hi = z.lo;
    return z;
}

// ---- 8-element loads and stores ------------------------------------------------

// W (fp32 or bf16) elements (r, c .. c+7) of an m x n row-major matrix, zero
// outside.  vec: n % 8 == 0, so the eight are either all inside or all outside.
template <typename TW>
__device__ __forceinline__ F8 load_w8(const TW* W, int m, int n, int r, int c, bool vec) {
    F8 v = zero8();
    if (r >= m || c >= n) return v;
    const int64_t idx = int64_t(r) * n + c;
    if (vec) {
        if constexpr (sizeof(TW) == 4) {
            v.lo = *reinterpret_cast<const float4*>(W + idx);
            v.hi = *reinterpret_cast<const float4*>(W + idx + 4);
        } else {
            const uint4 u = *reinterpret_cast<const uint4*>(W + idx);
            v.lo = make_float4(bf2f(u.x & 0xffff), bf2f(u.x >> 16), bf2f(u.y & 0xffff), bf2f(u.y >> 16));
            v.hi = make_float4(bf2f(u.z & 0xffff), bf2f(u.z >> 16), bf2f(u.w & 0xffff), bf2f(u.w >> 16));
        }
    } else {
        float t[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int e = 0; e < 8 && c + e < n; ++e) {
            if constexpr (sizeof(TW) == 4)
                t[e] = reinterpret_cast<const float*>(W)[idx + e];
            else
                t[e] = bf2f(reinterpret_cast<const uint16_t*>(W)[idx + e]);
        }
        v.lo = make_float4(t[0], t[1], t[2], t[3]);
        v.hi = make_float4(t[4], t[5], t[6], t[7]);
    }
    return v;
}

// Eight W elements at a 16-byte aligned offset (the flat tiles).
template <typename TW>
__device__ __forceinline__ F8 load_w8_at(const TW* W, int64_t idx) {
    F8 v;
    if constexpr (sizeof(TW) == 4) {
        v.lo = *reinterpret_cast<const float4*>(W + idx);
        v.hi = *reinterpret_cast<const float4*>(W + idx + 4);
    } else {
        const uint4 u = *reinterpret_cast<const uint4*>(W + idx);
        v.lo = make_float4(bf2f(u.x & 0xffff), bf2f(u.x >> 16), bf2f(u.y & 0xffff), bf2f(u.y >> 16));
        v.hi = make_float4(bf2f(u.z & 0xffff), bf2f(u.z >> 16), bf2f(u.w & 0xffff), bf2f(u.w >> 16));
    }
    return v;
}

__device__ __forceinline__ uint32_t pack_bf2(float a, float b) {
    return uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(a))) |
           (uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(b))) << 16);
}

// Eight elements at a 16-byte aligned offset.
template <typename TW>
__device__ __forceinline__ void store_w8_at(TW* W, int64_t idx, const F8& v) {
    if constexpr (sizeof(TW) == 4) {
        *reinterpret_cast<float4*>(W + idx) = v.lo;
        *reinterpret_cast<float4*>(W + idx + 4) = v.hi;
    } else {
        *reinterpret_cast<uint4*>(W + idx) = make_uint4(pack_bf2(v.lo.x, v.lo.y), pack_bf2(v.lo.z, v.lo.w),
                                                        pack_bf2(v.hi.x, v.hi.y), pack_bf2(v.hi.z, v.hi.w));
    }
}

template <typename TW>
__device__ __forceinline__ void store_w8(TW* W, int n, int r, int c, bool vec, const F8& v) {
    const int64_t idx = int64_t(r) * n + c;
    if (vec) {
        store_w8_at<TW>(W, idx, v);
    } else {
        const float t[8] = {v.lo.x, v.lo.y, v.lo.z, v.lo.w, v.hi.x, v.hi.y, v.hi.z, v.hi.w};
        for (int e = 0; e < 8 && c + e < n; ++e) {
            if constexpr (sizeof(TW) == 4)
                reinterpret_cast<float*>(W)[idx + e] = t[e];
            else
                reinterpret_cast<__nv_bfloat16*>(W)[idx + e] = __float2bfloat16_rn(t[e]);
        }
    }
}

// Iterate buffer elements [off .. off+7] (aligned: ld is a multiple of 64).
template <typename TX>
__device__ __forceinline__ F8 load_x8(const void* X, int64_t off) {
    F8 v;
    if constexpr (sizeof(TX) == 4) {
        const float* x = reinterpret_cast<const float*>(X) + off;
        v.lo = *reinterpret_cast<const float4*>(x);
        v.hi = *reinterpret_cast<const float4*>(x + 4);
    } else {
        const uint4 u = *reinterpret_cast<const uint4*>(reinterpret_cast<const uint16_t*>(X) + off);
        if constexpr (std::is_same<TX, __half>::value) {
            const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&u.x));
            const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&u.y));
            const float2 c = __half22float2(*reinterpret_cast<const __half2*>(&u.z));
            const float2 d = __half22float2(*reinterpret_cast<const __half2*>(&u.w));
            v.lo = make_float4(a.x, a.y, b.x, b.y);
            v.hi = make_float4(c.x, c.y, d.x, d.y);
        } else {
            v.lo = make_float4(bf2f(u.x & 0xffff), bf2f(u.x >> 16), bf2f(u.y & 0xffff), bf2f(u.y >> 16));
            v.hi = make_float4(bf2f(u.z & 0xffff), bf2f(u.z >> 16), bf2f(u.w & 0xffff), bf2f(u.w >> 16));
        }
    }
    return v;
}

template <typename TX>
__device__ __forceinline__ uint32_t pack_x2(float a, float b) {
    if constexpr (std::is_same<TX, __half>::value) {
        __half2 h = __floats2half2_rn(a, b);
        return *reinterpret_cast<uint32_t*>(&h);
    } else {
        return pack_bf2(a, b);
    }
}

template <typename TX>
__device__ __forceinline__ void store_x8(void* X, int64_t off, const F8& v) {
    if constexpr (sizeof(TX) == 4) {
        float* x = reinterpret_cast<float*>(X) + off;
        *reinterpret_cast<float4*>(x) = v.lo;
        *reinterpret_cast<float4*>(x + 4) = v.hi;
    } else {
        *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(X) + off) =
            make_uint4(pack_x2<TX>(v.lo.x, v.lo.y), pack_x2<TX>(v.lo.z, v.lo.w), pack_x2<TX>(v.hi.x, v.hi.y),
                       pack_x2<TX>(v.hi.z, v.hi.w));
    }
}

// bf16 hi/lo mode: the residuals v - bf16(v) of eight values.
__device__ __forceinline__ float bf_lo(float v) { return v - __bfloat162float(__float2bfloat16_rn(v)); }
__device__ __forceinline__ F8 lo8(const F8& v) {
    F8 r;
    r.lo = make_float4(bf_lo(v.lo.x), bf_lo(v.lo.y), bf_lo(v.lo.z), bf_lo(v.lo.w));
    r.hi = make_float4(bf_lo(v.hi.x), bf_lo(v.hi.y), bf_lo(v.hi.z), bf_lo(v.hi.w));
    return r;
}

__device__ __forceinline__ float dot8(const F8& a, const F8& b, float acc) {
    acc = fmaf(a.lo.x, b.lo.x, acc);
    acc = fmaf(a.lo.y, b.lo.y, acc);
    acc = fmaf(a.lo.z, b.lo.z, acc);
    acc = fmaf(a.lo.w, b.lo.w, acc);
    acc = fmaf(a.hi.x, b.hi.x, acc);
    acc = fmaf(a.hi.y, b.hi.y, acc);
    acc = fmaf(a.hi.z, b.hi.z, acc);
    acc = fmaf(a.hi.w, b.hi.w, acc);
    return acc;
}

// ---- reductions ----------------------------------------------------------------

__device__ __forceinline__ float block_sum(float v, float* red) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float s = 0.f;
    if (warp == 0) {
        s = lane < (kThreads / 32) ? red[lane] : 0.f;
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    }
    return s;  // valid in thread 0
}

// Block-wide sum and max of one value per thread: valid in thread 0.
__device__ __forceinline__ float2 block_sum_max(float v, float m) {
    __shared__ float rs[kThreads / 32], rm[kThreads / 32];
    for (int o = 16; o > 0; o >>= 1) {
        v += __shfl_xor_sync(0xffffffffu, v, o);
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        rs[warp] = v;
        rm[warp] = m;
    }
    __syncthreads();
    float2 r = make_float2(0.f, 0.f);
    if (warp == 0) {
        r.x = lane < (kThreads / 32) ? rs[lane] : 0.f;
        r.y = lane < (kThreads / 32) ? rm[lane] : 0.f;
        for (int o = 16; o > 0; o >>= 1) {
            r.x += __shfl_xor_sync(0xffffffffu, r.x, o);
            r.y = fmaxf(r.y, __shfl_xor_sync(0xffffffffu, r.y, o));
        }
    }
    return r;
}

__device__ __forceinline__ float absmax8(const F8& a, float m) {
    m = fmaxf(m, fmaxf(fmaxf(fabsf(a.lo.x), fabsf(a.lo.y)), fmaxf(fabsf(a.lo.z), fabsf(a.lo.w))));
    return fmaxf(m, fmaxf(fmaxf(fabsf(a.hi.x), fabsf(a.hi.y)), fmaxf(fabsf(a.hi.z), fabsf(a.hi.w))));
}

// An unscaled fp16 copy keeps every value of W at full relative precision
// and below overflow when max |w| <= 2^15, and its subnormal spacing (2^-24)
// costs no more than in the scaled X_0 when ||W||_F >= 1; bf16 has fp32's
// exponent range.
// bf16 keeps every unscaled copy (its exponent range is fp32's), so the
// re-cast below, which writes no low parts, never runs in bf16 hi/lo mode.
__device__ __forceinline__ bool unscaled_cast_ok(int elem, float maxabs, double frob) {
    return elem == kBF16 || maxabs == 0.f || (maxabs <= 32768.f && frob >= 1.0);
}

// Where this thread's 8-element group of row pass k lies: in a 2-D tile
// (row r0 + 4 k, columns c .. c + 7), or in a flat tile (elements e0 + 2048 k
// .. + 7 of W and, at the same offset, of the iterate buffer).
constexpr int kPassElems = kThreads * kMemVec;
struct Span {
    bool flat;
    int r0, c;   // 2-D: the thread's first row, its first column
    int64_t e0;  // flat: the thread's first element
};

__device__ __forceinline__ Span span_of(const MemItem& it) {
    Span t;
    t.flat = it.tile_r == kFlatTile;
    t.r0 = it.tile_r * kMemRows + int(threadIdx.x) / kVecPerRow;
    t.c = it.tile_c * kMemCols + (int(threadIdx.x) % kVecPerRow) * kMemVec;
    t.e0 = int64_t(it.seq) * (kMemRows * kMemCols) + int64_t(threadIdx.x) * kMemVec;
    return t;
}

// Pass k's group lies in W (all 8 elements in a flat tile, where n % 8 == 0;
// in a 2-D tile the row does, and the first column: the scalar paths mask
// the rest).
__device__ __forceinline__ bool in_w(const Span& t, const MatDev& md, int k) {
    if (t.flat) return t.e0 + int64_t(k) * kPassElems < int64_t(md.m) * md.n;
    return t.r0 + k * kRowsPerPass < md.m && t.c < md.n;
}

// Pass k's group lies in the (padded) iterate buffer.
__device__ __forceinline__ bool in_x(const Span& t, const MatDev& md, int k) {
    if (t.flat) return t.e0 + int64_t(k) * kPassElems < int64_t(md.rows) * md.ld;
    return t.r0 + k * kRowsPerPass < md.rows && t.c < md.ld;
}

__device__ __forceinline__ int64_t x_off(const Span& t, const MatDev& md, int k) {
    if (t.flat) return t.e0 + int64_t(k) * kPassElems;
    return int64_t(t.r0 + k * kRowsPerPass) * md.ld + t.c;
}

// W's (or a same-shaped gradient's) 8 elements of pass k, zero outside.
template <typename TW>
__device__ __forceinline__ F8 load_w(const TW* W, const MatDev& md, const Span& t, int k, bool vec) {
    if (t.flat) return in_w(t, md, k) ? load_w8_at<TW>(W, t.e0 + int64_t(k) * kPassElems) : zero8();
    return load_w8<TW>(W, md.m, md.n, t.r0 + k * kRowsPerPass, t.c, vec);
}

template <typename TW>
__device__ __forceinline__ void store_w(TW* W, const MatDev& md, const Span& t, int k, bool vec, const F8& v) {
    if (t.flat)
        store_w8_at<TW>(W, t.e0 + int64_t(k) * kPassElems, v);
    else
        store_w8<TW>(W, md.n, t.r0 + k * kRowsPerPass, t.c, vec, v);
}

// ---- kernels ---------------------------------------------------------------------

template <typename TW>
// Six blocks per SM (at most 40 registers a thread).
__global__ void __launch_bounds__(kThreads, 6) sumsq_kernel(const MemLaunch p) {
    ptx::griddep_wait();  // inputs come from the previous kernel (programmatic launch)
    ptx::griddep_launch_dependents();
    __shared__ float red[kThreads / 32];
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    const bool vec = (md.n & 7) == 0;
    const Span tc = span_of(it);
    F8 w[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) w[k] = load_w<TW>(W, md, tc, k, vec);
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < kPasses; ++k) acc = dot8(w[k], w[k], acc);
    const float part = block_sum(acc, red);
    if (threadIdx.x == 0) p.partials[p.tile_base[it.mat] + it.seq] = part;
}

// sumsq and cast in one read of W (16-bit iterates).  Items tile the padded
// buffer (rows x ld); the buffer receives W rounded to 16 bits, unscaled, and
// zeros in the padding; one partial of ||W||^2 and one of max |w| per item.
// In bf16 hi/lo mode (a low-part buffer xlo) the low parts w - bf16(w) too.
template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads, 4) normcast_kernel(const MemLaunch p) {
    ptx::griddep_wait();  // inputs come from the previous kernel (programmatic launch)
    ptx::griddep_launch_dependents();
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    void* X = md.x[p.cur];
    const bool vec = (md.n & 7) == 0;
    const Span tc = span_of(it);
    F8 w[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) w[k] = load_w<TW>(W, md, tc, k, vec);
#pragma unroll
    for (int k = 0; k < kPasses; ++k)
        if (in_x(tc, md, k)) store_x8<TX>(X, x_off(tc, md, k), w[k]);
    if constexpr (std::is_same<TX, __nv_bfloat16>::value) {
        void* XL = md.xlo[p.cur];
        if (XL != nullptr) {
#pragma unroll
            for (int k = 0; k < kPasses; ++k)
                if (in_x(tc, md, k)) store_x8<TX>(XL, x_off(tc, md, k), lo8(w[k]));
        }
    }
    float acc = 0.f, mx = 0.f;
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        acc = dot8(w[k], w[k], acc);
        mx = absmax8(w[k], mx);
    }
    const float2 sm = block_sum_max(acc, mx);
    if (threadIdx.x == 0) {
        p.partials[p.tile_base[it.mat] + it.seq] = sm.x;
        p.partials_max[p.tile_base[it.mat] + it.seq] = sm.y;
    }
}

// Items tile the padded buffer (rows x ld); zeros are written to the padding.
template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads) cast_kernel(const MemLaunch p) {
    ptx::griddep_wait();  // inputs come from the previous kernel (programmatic launch)
    ptx::griddep_launch_dependents();
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    void* X = md.x[p.cur];
    const bool vec = (md.n & 7) == 0;
    const Span tc = span_of(it);
    if (!tc.flat && tc.c >= md.ld) return;
    F8 w[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) w[k] = load_w<TW>(W, md, tc, k, vec);
    const float scale = p.scalars[it.mat].scale;
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        if (in_x(tc, md, k)) {
            F8 v;
            v.lo = make_float4(w[k].lo.x * scale, w[k].lo.y * scale, w[k].lo.z * scale, w[k].lo.w * scale);
            v.hi = make_float4(w[k].hi.x * scale, w[k].hi.y * scale, w[k].hi.z * scale, w[k].hi.w * scale);
            store_x8<TX>(X, x_off(tc, md, k), v);
        }
    }
}

template <typename TW, typename TX>
// At most 64 registers a thread, so that four blocks share an SM: with three
// (68 registers) the pass reached 0.69 of the measured HBM bandwidth on the
// ViT-L/16 set, with four it is 11% faster.
__global__ void __launch_bounds__(kThreads, 4) dot_kernel(const MemLaunch p) {
    ptx::griddep_wait();  // inputs come from the previous kernel (programmatic launch)
    ptx::griddep_launch_dependents();
    __shared__ float red[kThreads / 32];
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    const void* X = md.x[p.cur];
    float acc = 0.f;
    if (it.tile_r == kFlatTile) {
        // flat tile: W and X_T at the same offsets
        const int64_t e0 = int64_t(it.seq) * (kMemRows * kMemCols) + int64_t(threadIdx.x) * kMemVec;
        const int64_t total = int64_t(md.m) * md.n;
        F8 w[kPasses], x[kPasses];
#pragma unroll
        for (int k = 0; k < kPasses; ++k) {
            const int64_t e = e0 + int64_t(k) * kPassElems;
            w[k] = e < total ? load_w8_at<TW>(W, e) : zero8();
            x[k] = e < total ? load_x8<TX>(X, e) : zero8();
        }
#pragma unroll
        for (int k = 0; k < kPasses; ++k) acc = dot8(w[k], x[k], acc);
    } else {
        const bool vec = (md.n & 7) == 0;
        const Span tc = span_of(it);
        F8 w[kPasses], x[kPasses];
#pragma unroll
        for (int k = 0; k < kPasses; ++k) {
            w[k] = load_w<TW>(W, md, tc, k, vec);
            x[k] = in_w(tc, md, k) ? load_x8<TX>(X, x_off(tc, md, k)) : zero8();
        }
#pragma unroll
        for (int k = 0; k < kPasses; ++k) acc = dot8(w[k], x[k], acc);
    }
    const float part = block_sum(acc, red);
    if (threadIdx.x == 0) p.partials[p.tile_base[it.mat] + it.seq] = part;
}

// Values L_i and the loss lambda * sum_i L_i, by one whole block: thread t
// handles matrices t, t + 128, ...; the partial sums are combined in a fixed
// tree, so the result does not depend on timing.
__device__ void finalize_loss(const MemLaunch& p) {
    __shared__ double red[4];
    const double eps = static_cast<double>(p.eps);
    double part = 0.0;
    for (int i = threadIdx.x; i < p.count; i += 128) {
        const double n_i = __ldcg(&p.scalars[i].n_hat);
        double L;
        if (p.variant == 0) {
            const double fr = sqrt(__ldcg(&p.scalars[i].frob_sq)) + eps;
            const double reg = n_i / fr;
            L = reg * reg;
        } else {
            L = n_i;
        }
        if (p.per_matrix_out) p.per_matrix_out[i] = static_cast<float>(L);
        part += L;
    }
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
    __syncthreads();
    if (threadIdx.x == 0)
        *p.loss_out = static_cast<float>(static_cast<double>(p.lambda) * ((red[0] + red[1]) + (red[2] + red[3])));
}

// Thread 0 of the block of matrix `mat`: stores the sum and the derived
// coefficients; returns true in the last block to finish the n_hat pass.
__device__ bool finalize_matrix(const MemLaunch& p, int which, int mat, double tot) {
    MatScalars& sc = p.scalars[mat];
    const double eps = static_cast<double>(p.eps);
    if (which == 0) {
        sc.frob_sq = tot;
        sc.scale = static_cast<float>(1.0 / (sqrt(tot) + eps));
        sc.x0_scale = 1.f;
        if (!isfinite(tot)) atomicOr(p.status, kStatusNonFinite);
        return false;
    }
    sc.n_hat = tot;
    const double frob = sqrt(sc.frob_sq) + eps;
    const double lg = static_cast<double>(p.lambda) * static_cast<double>(p.grad_scale);
    double alpha, beta;
    if (p.variant == 0) {
        const double reg = tot / frob;
        alpha = lg * 2.0 * reg / frob;
        beta = lg * 2.0 * reg * tot / (frob * frob * frob);
    } else {
        alpha = lg;
        beta = 0.0;
    }
    const bool bad = !isfinite(tot) || !isfinite(alpha) || !isfinite(beta);
    sc.alpha = static_cast<float>(alpha);
    sc.beta = static_cast<float>(beta);
    sc.skip = bad ? 1 : 0;
    if (bad) atomicOr(p.status, kStatusNonFinite);
    __threadfence();
    if (atomicAdd(p.counters + p.count, 1u) != static_cast<uint32_t>(p.count - 1)) return false;
    p.counters[p.count] = 0u;  // leave the counter clean for the next call
    __threadfence();
    return true;
}

// One block per matrix: adds the matrix's tile partials in index order (double)
// and derives the per-matrix coefficients the next pass needs.
//   which = 0: ||W||_F^2 and the cast scale 1 / (||W||_F + eps);
//   which = 2: the same after normcast, and x0_scale: the scale when the
//              unscaled copy is kept, else 1 after this block re-casts
//              X_0 = scale * W;
//   which = 1: n_hat and the gradient coefficients (Listing 1 backward times
//              lambda * grad_scale): Hoyer alpha = 2 reg / frob,
//              beta = 2 reg n_hat / frob^3 with reg = n_hat / frob; Nuc alpha = 1.
//              The last block to finish also writes the values L_i and the loss
//              lambda * sum_i L_i (finalize_loss).
__global__ void __launch_bounds__(128) finalize_kernel(const MemLaunch p, int which) {
    ptx::griddep_wait();  // inputs come from the previous kernel (programmatic launch)
    ptx::griddep_launch_dependents();
    __shared__ double red[4];
    __shared__ float redm[4];
    __shared__ int is_last;
    const int mat = blockIdx.x;
    const int base = p.tile_base[mat], n = p.tile_count[mat];
    const bool fused = which == 2;
    double s = 0.0;
    float m = 0.f;
    for (int i = threadIdx.x; i < n; i += 128) {
        s += static_cast<double>(__ldcg(p.partials + base + i));
        if (fused) m = fmaxf(m, __ldcg(p.partials_max + base + i));
    }
    for (int o = 16; o > 0; o >>= 1) {
        s += __shfl_xor_sync(0xffffffffu, s, o);
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    }
    if ((threadIdx.x & 31) == 0) {
        red[threadIdx.x >> 5] = s;
        redm[threadIdx.x >> 5] = m;
    }
    __syncthreads();
    const double tot = (red[0] + red[1]) + (red[2] + red[3]);
    if (!fused) {
        if (threadIdx.x == 0) is_last = finalize_matrix(p, which, mat, tot) ? 1 : 0;
        __syncthreads();
        if (is_last) finalize_loss(p);
        return;
    }
    // after normcast: keep the unscaled copy (x0_scale = scale) or re-cast it
    const float mx = fmaxf(fmaxf(redm[0], redm[1]), fmaxf(redm[2], redm[3]));
    const double fr = sqrt(tot);
    const float scale = static_cast<float>(1.0 / (fr + static_cast<double>(p.eps)));
    const bool ok = unscaled_cast_ok(p.elem, mx, fr);
    if (threadIdx.x == 0) {
        MatScalars& sc = p.scalars[mat];
        sc.frob_sq = tot;
        sc.scale = scale;
        sc.x0_scale = ok ? scale : 1.f;
        if (!isfinite(tot)) atomicOr(p.status, kStatusNonFinite);
    }
    if (ok) return;
    // X_0 = scale * W over W's region (the padding already holds zeros)
    const MatDev md = p.mats[mat];
    const void* W = p.weights[mat];
    const int64_t total = int64_t(md.m) * md.n;
    for (int64_t i = threadIdx.x; i < total; i += 128) {
        const int64_t r = i / md.n, c = i - r * md.n;
        const float w = p.wdtype == 0 ? reinterpret_cast<const float*>(W)[i]
                                      : bf2f(reinterpret_cast<const uint16_t*>(W)[i]);
        const int64_t o = r * md.ld + c;
        if (p.elem == kF16)
            reinterpret_cast<__half*>(md.x[p.cur])[o] = __float2half_rn(w * scale);
        else
            reinterpret_cast<__nv_bfloat16*>(md.x[p.cur])[o] = __float2bfloat16_rn(w * scale);
    }
}

template <typename TW, typename TX>
// Loads for two of the four row passes at a time: with all four in flight a
// thread needs 128 registers (two blocks per SM); in halves it fits four
// blocks per SM, 20% faster on the ViT-L/16 set.
__global__ void __launch_bounds__(kThreads, 4) combine_kernel(const MemLaunch p) {
    ptx::griddep_wait();  // inputs come from the previous kernel (programmatic launch)
    ptx::griddep_launch_dependents();
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const Span tc = span_of(it);
    const MatScalars& sc = p.scalars[it.mat];
    if (sc.skip || (!tc.flat && tc.c >= md.n)) return;  // non-finite: leave the gradient untouched
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    TW* G = reinterpret_cast<TW*>(p.grads[it.mat]);
    const void* X = md.x[p.cur];
    const float fa = sc.alpha, fb = sc.beta;
    const bool vec = (md.n & 7) == 0;
#pragma unroll
    for (int h = 0; h < kPasses; h += 2) {
        F8 w[2], x[2], g[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            w[q] = load_w<TW>(W, md, tc, h + q, vec);
            if (p.out_mode == kOutAccumulate) g[q] = load_w<TW>(G, md, tc, h + q, vec);
            else if (p.out_mode == kOutDescent) g[q] = w[q];  // G points at W: applied in place
            else g[q] = zero8();
            x[q] = in_w(tc, md, h + q) ? load_x8<TX>(X, x_off(tc, md, h + q)) : zero8();
        }
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            if (!in_w(tc, md, h + q)) continue;
            F8 o;
            o.lo.x = g[q].lo.x + (fa * x[q].lo.x - fb * w[q].lo.x);
            o.lo.y = g[q].lo.y + (fa * x[q].lo.y - fb * w[q].lo.y);
            o.lo.z = g[q].lo.z + (fa * x[q].lo.z - fb * w[q].lo.z);
            o.lo.w = g[q].lo.w + (fa * x[q].lo.w - fb * w[q].lo.w);
            o.hi.x = g[q].hi.x + (fa * x[q].hi.x - fb * w[q].hi.x);
            o.hi.y = g[q].hi.y + (fa * x[q].hi.y - fb * w[q].hi.y);
            o.hi.z = g[q].hi.z + (fa * x[q].hi.z - fb * w[q].hi.z);
            o.hi.w = g[q].hi.w + (fa * x[q].hi.w - fb * w[q].hi.w);
            store_w<TW>(G, md, tc, h + q, vec, o);
        }
    }
}

}  // namespace

cudaError_t launch_sumsq(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    if (p.wdtype == 0) return launch_kernel(sumsq_kernel<float>, p.num_items, kThreads, 0, s, p.pdl != 0, p);
    return launch_kernel(sumsq_kernel<__nv_bfloat16>, p.num_items, kThreads, 0, s, p.pdl != 0, p);
}

#define SLORR_LAUNCH_WX(KERNEL, TW, TX) launch_kernel(KERNEL<TW, TX>, p.num_items, kThreads, 0, s, p.pdl != 0, p)
#define SLORR_DISPATCH_WX(KERNEL)                                                                  \
    do {                                                                                           \
        if (p.wdtype == 0) {                                                                       \
            if (p.elem == kF32) return SLORR_LAUNCH_WX(KERNEL, float, float);                      \
            if (p.elem == kF16) return SLORR_LAUNCH_WX(KERNEL, float, __half);                     \
            return SLORR_LAUNCH_WX(KERNEL, float, __nv_bfloat16);                                  \
        }                                                                                          \
        if (p.elem == kF32) return SLORR_LAUNCH_WX(KERNEL, __nv_bfloat16, float);                  \
        if (p.elem == kF16) return SLORR_LAUNCH_WX(KERNEL, __nv_bfloat16, __half);                 \
        return SLORR_LAUNCH_WX(KERNEL, __nv_bfloat16, __nv_bfloat16);                              \
    } while (0)

cudaError_t launch_cast(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    SLORR_DISPATCH_WX(cast_kernel);
}

cudaError_t launch_dot(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    SLORR_DISPATCH_WX(dot_kernel);
}

cudaError_t launch_normcast(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    if (p.elem == kF32) return cudaErrorInvalidValue;  // 16-bit iterates only
    SLORR_DISPATCH_WX(normcast_kernel);
}

cudaError_t launch_finalize(const MemLaunch& p, int which, cudaStream_t s) {
    return launch_kernel(finalize_kernel, p.count, 128, 0, s, p.pdl != 0, p, which);
}

// One thread: out = sum of the n partial losses in index order (double).
__global__ void sum_parts_kernel(const float* __restrict__ parts, int n, float* __restrict__ out) {
    ptx::griddep_wait();
    ptx::griddep_launch_dependents();
    if (threadIdx.x == 0 && blockIdx.x == 0) {
        double t = 0.0;
        for (int i = 0; i < n; ++i) t += static_cast<double>(parts[i]);
        *out = static_cast<float>(t);
    }
}

cudaError_t launch_sum_parts(const float* parts, int n, float* out, cudaStream_t s) {
    return launch_kernel(sum_parts_kernel, 1, 32, 0, s, false, parts, n, out);
}

cudaError_t launch_combine(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    SLORR_DISPATCH_WX(combine_kernel);
}

}  // namespace slorr
