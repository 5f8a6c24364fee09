// Memory-bound passes of the SLORR hot path, grouped over all weight matrices:
//   sumsq   ||W_i||_F^2                                  (Listing 1, frob)
//   cast    X_0 = W_i / (||W_i||_F + eps), zero padded    (Sec. 3 "Computing the polar factor")
//   dot     n_hat_i = sum(W_i * P_hat_i), values L_i and the loss
//                                                        (Sec. 3 "Computing the nuclear ...", Listing 1)
//   combine W_i.grad += lambda * grad_scale * G_i       (Listing 1 backward, Alg. 2)
// The iterates are stored in W's orientation (row-major, row length `ld`), so
// every pass is elementwise.  A block handles one kMemRows x kMemCols tile:
// each of its 256 threads owns 4 consecutive columns of 8 rows and issues all
// eight 128-bit loads before using them (64-bit for 16-bit data).  Rows whose
// length is not a multiple of 4 take a scalar path.  Cross-tile sums are
// deterministic: each block writes a partial; the last block of a matrix (per-
// matrix counter) adds the partials in index order in double precision.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "internal.h"

namespace slorr {
namespace {

constexpr int kThreads = 256;
constexpr int kVecPerRow = kMemCols / 4;             // 128 threads per tile row
constexpr int kRowsPerPass = kThreads / kVecPerRow;  // 2
constexpr int kPasses = kMemRows / kRowsPerPass;     // 8

__device__ __forceinline__ float bf2f(uint16_t u) { return __uint_as_float(uint32_t(u) << 16); }

// ---- 4-element loads and stores ------------------------------------------------

// W (fp32 or bf16) elements (r, c .. c+3) of an m x n row-major matrix, zero
// outside.  vec: n % 4 == 0, so the four are either all inside or all outside.
template <typename TW>
__device__ __forceinline__ float4 load_w4(const TW* W, int m, int n, int r, int c, bool vec) {
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r >= m || c >= n) return v;
    const int64_t idx = int64_t(r) * n + c;
    if (vec) {
        if constexpr (sizeof(TW) == 4) {
            v = *reinterpret_cast<const float4*>(W + idx);
        } else {
            const uint2 u = *reinterpret_cast<const uint2*>(W + idx);
            v = make_float4(bf2f(u.x & 0xffff), bf2f(u.x >> 16), bf2f(u.y & 0xffff), bf2f(u.y >> 16));
        }
    } else {
        float t[4] = {0.f, 0.f, 0.f, 0.f};
        for (int e = 0; e < 4 && c + e < n; ++e) {
            if constexpr (sizeof(TW) == 4)
                t[e] = reinterpret_cast<const float*>(W)[idx + e];
            else
                t[e] = bf2f(reinterpret_cast<const uint16_t*>(W)[idx + e]);
        }
        v = make_float4(t[0], t[1], t[2], t[3]);
    }
    return v;
}

template <typename TW>
__device__ __forceinline__ void store_w4(TW* W, int n, int r, int c, bool vec, float4 v) {
    const int64_t idx = int64_t(r) * n + c;
    if (vec) {
        if constexpr (sizeof(TW) == 4) {
            *reinterpret_cast<float4*>(W + idx) = v;
        } else {
            const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(v.x)) |
                                (uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(v.y))) << 16);
            const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(v.z)) |
                                (uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(v.w))) << 16);
            *reinterpret_cast<uint2*>(W + idx) = make_uint2(lo, hi);
        }
    } else {
        const float t[4] = {v.x, v.y, v.z, v.w};
        for (int e = 0; e < 4 && c + e < n; ++e) {
            if constexpr (sizeof(TW) == 4)
                reinterpret_cast<float*>(W)[idx + e] = t[e];
            else
                reinterpret_cast<__nv_bfloat16*>(W)[idx + e] = __float2bfloat16_rn(t[e]);
        }
    }
}

// Iterate buffer elements [off .. off+3] (aligned: ld is a multiple of 64).
template <typename TX>
__device__ __forceinline__ float4 load_x4(const void* X, int64_t off) {
    if constexpr (sizeof(TX) == 4) {
        return *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(X) + off);
    } else {
        const uint2 u = *reinterpret_cast<const uint2*>(reinterpret_cast<const uint16_t*>(X) + off);
        if constexpr (std::is_same<TX, __half>::value) {
            const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&u.x));
            const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&u.y));
            return make_float4(a.x, a.y, b.x, b.y);
        } else {
            return make_float4(bf2f(u.x & 0xffff), bf2f(u.x >> 16), bf2f(u.y & 0xffff), bf2f(u.y >> 16));
        }
    }
}

template <typename TX>
__device__ __forceinline__ void store_x4(void* X, int64_t off, float4 v) {
    if constexpr (sizeof(TX) == 4) {
        *reinterpret_cast<float4*>(reinterpret_cast<float*>(X) + off) = v;
    } else if constexpr (std::is_same<TX, __half>::value) {
        __half2 a = __floats2half2_rn(v.x, v.y), b = __floats2half2_rn(v.z, v.w);
        *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(X) + off) =
            make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
    } else {
        __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
        *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(X) + off) =
            make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
    }
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

// Deterministic sum of partials[base .. base+n) by warp 0, in double.
__device__ __forceinline__ double sum_partials(const float* partials, int base, int n) {
    double s = 0.0;
    const int lane = threadIdx.x & 31;
    for (int i = lane; i < n; i += 32) s += static_cast<double>(__ldcg(partials + base + i));
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    return s;
}

// Publishes this block's partial; true (in every thread) in the block that
// completed the matrix.
__device__ __forceinline__ bool finish_tile(const MemLaunch& p, int mat, int seq, float part,
                                            int* flag_smem) {
    if (threadIdx.x == 0) {
        p.partials[p.tile_base[mat] + seq] = part;
        __threadfence();
        const uint32_t done = atomicAdd(p.counters + mat, 1u);
        const bool last = done == static_cast<uint32_t>(p.tile_count[mat] - 1);
        if (last) {
            p.counters[mat] = 0u;  // leave the counter clean for the next call
            __threadfence();
        }
        *flag_smem = last ? 1 : 0;
    }
    __syncthreads();
    return *flag_smem != 0;
}

struct TileCoord {
    int r0, c;  // first row of this thread, its first column
};

__device__ __forceinline__ TileCoord tile_coord(const MemItem& it) {
    TileCoord t;
    t.r0 = it.tile_r * kMemRows + int(threadIdx.x) / kVecPerRow;
    t.c = it.tile_c * kMemCols + (int(threadIdx.x) % kVecPerRow) * 4;
    return t;
}

// ---- kernels ---------------------------------------------------------------------

template <typename TW>
__global__ void __launch_bounds__(kThreads) sumsq_kernel(const MemLaunch p) {
    __shared__ float red[kThreads / 32];
    __shared__ int flag;
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    const bool vec = (md.n & 3) == 0;
    const TileCoord tc = tile_coord(it);
    float4 w[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) w[k] = load_w4<TW>(W, md.m, md.n, tc.r0 + k * kRowsPerPass, tc.c, vec);
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        acc = fmaf(w[k].x, w[k].x, acc);
        acc = fmaf(w[k].y, w[k].y, acc);
        acc = fmaf(w[k].z, w[k].z, acc);
        acc = fmaf(w[k].w, w[k].w, acc);
    }
    const float part = block_sum(acc, red);
    if (finish_tile(p, it.mat, it.seq, part, &flag) && threadIdx.x < 32) {
        const double s = sum_partials(p.partials, p.tile_base[it.mat], p.tile_count[it.mat]);
        if (threadIdx.x == 0) {
            p.scalars[it.mat].frob_sq = s;
            if (!isfinite(s)) atomicOr(p.status, kStatusNonFinite);
        }
    }
}

// Items tile the padded buffer (rows x ld); zeros are written to the padding.
template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads) cast_kernel(const MemLaunch p) {
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    const double f = sqrt(p.scalars[it.mat].frob_sq);
    const float scale = static_cast<float>(1.0 / (f + static_cast<double>(p.eps)));
    void* X = md.x[p.cur];
    const bool vec = (md.n & 3) == 0;
    const TileCoord tc = tile_coord(it);
    if (tc.c >= md.ld) return;
    float4 w[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) w[k] = load_w4<TW>(W, md.m, md.n, tc.r0 + k * kRowsPerPass, tc.c, vec);
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        const int r = tc.r0 + k * kRowsPerPass;
        if (r < md.rows) {
            const float4 v = make_float4(w[k].x * scale, w[k].y * scale, w[k].z * scale, w[k].w * scale);
            store_x4<TX>(X, int64_t(r) * md.ld + tc.c, v);
        }
    }
}

template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads) dot_kernel(const MemLaunch p) {
    __shared__ float red[kThreads / 32];
    __shared__ int flag;
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    const void* X = md.x[p.cur];
    const bool vec = (md.n & 3) == 0;
    const TileCoord tc = tile_coord(it);
    float4 w[kPasses], x[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        const int r = tc.r0 + k * kRowsPerPass;
        w[k] = load_w4<TW>(W, md.m, md.n, r, tc.c, vec);
        x[k] = (r < md.m && tc.c < md.n) ? load_x4<TX>(X, int64_t(r) * md.ld + tc.c)
                                          : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        acc = fmaf(w[k].x, x[k].x, acc);
        acc = fmaf(w[k].y, x[k].y, acc);
        acc = fmaf(w[k].z, x[k].z, acc);
        acc = fmaf(w[k].w, x[k].w, acc);
    }
    const float part = block_sum(acc, red);
    if (!finish_tile(p, it.mat, it.seq, part, &flag)) return;
    if (threadIdx.x >= 32) return;
    const double nh = sum_partials(p.partials, p.tile_base[it.mat], p.tile_count[it.mat]);
    if (threadIdx.x == 0) {
        p.scalars[it.mat].n_hat = nh;
        if (!isfinite(nh)) atomicOr(p.status, kStatusNonFinite);
        // The last matrix to finish writes the values and the loss in index order.
        __threadfence();
        const uint32_t done = atomicAdd(p.counters + p.count, 1u);
        if (done == static_cast<uint32_t>(p.count - 1)) {
            p.counters[p.count] = 0u;
            __threadfence();
            double loss = 0.0;
            for (int i = 0; i < p.count; ++i) {
                const double n_i = __ldcg(&p.scalars[i].n_hat);
                double L;
                if (p.variant == 0) {
                    const double frob = sqrt(__ldcg(&p.scalars[i].frob_sq)) + static_cast<double>(p.eps);
                    const double reg = n_i / frob;
                    L = reg * reg;
                } else {
                    L = n_i;
                }
                if (p.per_matrix_out) p.per_matrix_out[i] = static_cast<float>(L);
                loss += L;
            }
            *p.loss_out = static_cast<float>(static_cast<double>(p.lambda) * loss);
        }
    }
}

template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads) combine_kernel(const MemLaunch p) {
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const TW* W = reinterpret_cast<const TW*>(p.weights[it.mat]);
    TW* G = reinterpret_cast<TW*>(p.grads[it.mat]);
    const void* X = md.x[p.cur];
    const double nh = p.scalars[it.mat].n_hat;
    const double frob = sqrt(p.scalars[it.mat].frob_sq) + static_cast<double>(p.eps);
    const double lg = static_cast<double>(p.lambda) * static_cast<double>(p.grad_scale);
    double alpha, beta;
    if (p.variant == 0) {  // 2 reg (P_hat / frob - n_hat / frob^3 W)
        const double reg = nh / frob;
        alpha = lg * 2.0 * reg / frob;
        beta = lg * 2.0 * reg * nh / (frob * frob * frob);
    } else {               // P_hat
        alpha = lg;
        beta = 0.0;
    }
    if (!isfinite(alpha) || !isfinite(beta)) {
        if (threadIdx.x == 0) atomicOr(p.status, kStatusNonFinite);
        return;  // leave this matrix's gradient untouched
    }
    const float fa = static_cast<float>(alpha), fb = static_cast<float>(beta);
    const bool vec = (md.n & 3) == 0;
    const TileCoord tc = tile_coord(it);
    if (tc.c >= md.n) return;
    float4 w[kPasses], x[kPasses], g[kPasses];
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        const int r = tc.r0 + k * kRowsPerPass;
        w[k] = load_w4<TW>(W, md.m, md.n, r, tc.c, vec);
        g[k] = load_w4<TW>(G, md.m, md.n, r, tc.c, vec);
        x[k] = r < md.m ? load_x4<TX>(X, int64_t(r) * md.ld + tc.c) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int k = 0; k < kPasses; ++k) {
        const int r = tc.r0 + k * kRowsPerPass;
        if (r >= md.m) continue;
        float4 o;
        o.x = g[k].x + (fa * x[k].x - fb * w[k].x);
        o.y = g[k].y + (fa * x[k].y - fb * w[k].y);
        o.z = g[k].z + (fa * x[k].z - fb * w[k].z);
        o.w = g[k].w + (fa * x[k].w - fb * w[k].w);
        store_w4<TW>(G, md.n, r, tc.c, vec, o);
    }
}

}  // namespace

cudaError_t launch_sumsq(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    if (p.wdtype == 0)
        sumsq_kernel<float><<<p.num_items, kThreads, 0, s>>>(p);
    else
        sumsq_kernel<__nv_bfloat16><<<p.num_items, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

#define SLORR_DISPATCH_WX(KERNEL)                                                                  \
    do {                                                                                           \
        if (p.wdtype == 0) {                                                                       \
            if (p.elem == kF32) KERNEL<float, float><<<p.num_items, kThreads, 0, s>>>(p);          \
            else if (p.elem == kF16) KERNEL<float, __half><<<p.num_items, kThreads, 0, s>>>(p);    \
            else KERNEL<float, __nv_bfloat16><<<p.num_items, kThreads, 0, s>>>(p);                \
        } else {                                                                                   \
            if (p.elem == kF32) KERNEL<__nv_bfloat16, float><<<p.num_items, kThreads, 0, s>>>(p);  \
            else if (p.elem == kF16) KERNEL<__nv_bfloat16, __half><<<p.num_items, kThreads, 0, s>>>(p); \
            else KERNEL<__nv_bfloat16, __nv_bfloat16><<<p.num_items, kThreads, 0, s>>>(p);        \
        }                                                                                          \
    } while (0)

cudaError_t launch_cast(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    SLORR_DISPATCH_WX(cast_kernel);
    return cudaGetLastError();
}

cudaError_t launch_dot(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    SLORR_DISPATCH_WX(dot_kernel);
    return cudaGetLastError();
}

cudaError_t launch_combine(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    SLORR_DISPATCH_WX(combine_kernel);
    return cudaGetLastError();
}

}  // namespace slorr
