// Memory-bound passes of the SLORR hot path, grouped over all weight matrices:
//   sumsq   ||W_i||_F^2                                  (Listing 1, frob)
//   cast    X_0 = W_i / (||W_i||_F + eps), Gram-side orientation, zero padded
//                                                        (Sec. 3 "Computing the polar factor")
//   dot     n_hat_i = sum(W_i * P_hat_i), values L_i and the loss
//                                                        (Sec. 3 "Computing the nuclear ...", Listing 1)
//   combine W_i.grad += lambda * grad_scale * G_i       (Listing 1 backward, Alg. 2)
// Each block handles one 64 x 64 tile.  Cross-tile sums are deterministic: a
// block writes its partial, the last block of a matrix (per-matrix counter)
// adds the partials in index order in double precision.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "internal.h"

namespace slorr {
namespace {

constexpr int kTile = 64;
constexpr int kThreads = 256;
constexpr int kRowsPerPass = kThreads / kTile;  // 4

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__half>(__half v) { return __half2float(v); }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __half from_f<__half>(float v) { return __float2half_rn(v); }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

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

// Publishes this block's partial and returns true in the block that completed
// the matrix (all threads see the result).
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

template <typename TW>
__device__ __forceinline__ float load_w(const void* base, int64_t idx) {
    return to_f<TW>(reinterpret_cast<const TW*>(base)[idx]);
}

// ---- sumsq ----------------------------------------------------------------------

template <typename TW>
__global__ void __launch_bounds__(kThreads) sumsq_kernel(const MemLaunch p) {
    __shared__ float red[kThreads / 32];
    __shared__ int flag;
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const void* W = p.weights[it.mat];
    const int c = it.tile_c * kTile + (threadIdx.x % kTile);
    const int r0 = it.tile_r * kTile + (threadIdx.x / kTile);
    float acc = 0.f;
    if (c < md.n) {
#pragma unroll 4
        for (int k = 0; k < kTile / kRowsPerPass; ++k) {
            const int r = r0 + k * kRowsPerPass;
            if (r < md.m) {
                const float w = load_w<TW>(W, static_cast<int64_t>(r) * md.n + c);
                acc = fmaf(w, w, acc);
            }
        }
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

// ---- cast -----------------------------------------------------------------------

// Items tile the padded iterate (Ppad x Qpad); writes X_0 including zeros in
// the padding.
template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads) cast_kernel(const MemLaunch p) {
    __shared__ float tile[kTile][kTile + 1];
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const void* W = p.weights[it.mat];
    const double f = sqrt(p.scalars[it.mat].frob_sq);
    const float scale = static_cast<float>(1.0 / (f + static_cast<double>(p.eps)));
    TX* X = reinterpret_cast<TX*>(md.x[p.cur]);
    const int p0 = it.tile_r * kTile, q0 = it.tile_c * kTile;
    const int lx = threadIdx.x % kTile, ly = threadIdx.x / kTile;
    if (!md.transposed) {
        // X[p][q] = W[p][q]
        for (int k = 0; k < kTile / kRowsPerPass; ++k) {
            const int pp = p0 + ly + k * kRowsPerPass, qq = q0 + lx;
            float v = 0.f;
            if (pp < md.P && qq < md.Q) v = load_w<TW>(W, static_cast<int64_t>(pp) * md.n + qq) * scale;
            X[static_cast<int64_t>(pp) * md.Qpad + qq] = from_f<TX>(v);
        }
    } else {
        // X[p][q] = W[q][p]: read W rows q (contiguous in p), write X rows p.
        for (int k = 0; k < kTile / kRowsPerPass; ++k) {
            const int qq = q0 + ly + k * kRowsPerPass, pp = p0 + lx;
            float v = 0.f;
            if (pp < md.P && qq < md.Q) v = load_w<TW>(W, static_cast<int64_t>(qq) * md.n + pp);
            tile[ly + k * kRowsPerPass][lx] = v;
        }
        __syncthreads();
        for (int k = 0; k < kTile / kRowsPerPass; ++k) {
            const int pl = ly + k * kRowsPerPass;
            const int pp = p0 + pl, qq = q0 + lx;
            X[static_cast<int64_t>(pp) * md.Qpad + qq] = from_f<TX>(tile[lx][pl] * scale);
        }
    }
}

// ---- W-tile traversal with the final iterate in W's orientation ---------------

// Loads, for this thread's 16 elements (rows r0 + ly + 4k, column c), the value
// of P_hat = X_T in W's orientation into xv[k].
template <typename TX>
__device__ __forceinline__ void load_phat(const MatDev& md, const TX* X, int r_base, int c_base,
                                          float (*tile)[kTile + 1], float xv[16]) {
    const int lx = threadIdx.x % kTile, ly = threadIdx.x / kTile;
    if (!md.transposed) {
        const int c = c_base + lx;
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int r = r_base + ly + k * kRowsPerPass;
            xv[k] = (r < md.m && c < md.n) ? to_f<TX>(X[static_cast<int64_t>(r) * md.Qpad + c]) : 0.f;
        }
    } else {
        // W(r, c) = X[c][r]: stage X rows c (contiguous in r) through shared memory.
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const int cl = ly + k * kRowsPerPass;
            const int c = c_base + cl, r = r_base + lx;
            tile[cl][lx] = (r < md.m && c < md.n) ? to_f<TX>(X[static_cast<int64_t>(c) * md.Qpad + r]) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < 16; ++k) xv[k] = tile[lx][ly + k * kRowsPerPass];
    }
}

template <typename TW, typename TX>
__global__ void __launch_bounds__(kThreads) dot_kernel(const MemLaunch p) {
    __shared__ float tile[kTile][kTile + 1];
    __shared__ float red[kThreads / 32];
    __shared__ int flag;
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const void* W = p.weights[it.mat];
    const TX* X = reinterpret_cast<const TX*>(md.x[p.cur]);
    const int r_base = it.tile_r * kTile, c_base = it.tile_c * kTile;
    float xv[16];
    load_phat<TX>(md, X, r_base, c_base, tile, xv);
    const int c = c_base + threadIdx.x % kTile;
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const int r = r_base + threadIdx.x / kTile + k * kRowsPerPass;
        if (r < md.m && c < md.n) acc = fmaf(load_w<TW>(W, static_cast<int64_t>(r) * md.n + c), xv[k], acc);
    }
    const float part = block_sum(acc, red);
    if (!finish_tile(p, it.mat, it.seq, part, &flag)) return;
    if (threadIdx.x >= 32) return;
    const double nh = sum_partials(p.partials, p.tile_base[it.mat], p.tile_count[it.mat]);
    if (threadIdx.x == 0) {
        p.scalars[it.mat].n_hat = nh;
        if (!isfinite(nh)) atomicOr(p.status, kStatusNonFinite);
        // Last matrix to finish writes the values and the loss in index order.
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
    __shared__ float tile[kTile][kTile + 1];
    const MemItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const void* W = p.weights[it.mat];
    void* G = p.grads[it.mat];
    const TX* X = reinterpret_cast<const TX*>(md.x[p.cur]);
    const double nh = p.scalars[it.mat].n_hat;
    const double frob = sqrt(p.scalars[it.mat].frob_sq) + static_cast<double>(p.eps);
    const double lg = static_cast<double>(p.lambda) * static_cast<double>(p.grad_scale);
    double alpha, beta;
    if (p.variant == 0) {
        const double reg = nh / frob;
        alpha = lg * 2.0 * reg / frob;
        beta = lg * 2.0 * reg * nh / (frob * frob * frob);
    } else {
        alpha = lg;
        beta = 0.0;
    }
    if (!isfinite(alpha) || !isfinite(beta)) {
        if (threadIdx.x == 0) atomicOr(p.status, kStatusNonFinite);
        return;  // leave this matrix's gradient untouched
    }
    const float fa = static_cast<float>(alpha), fb = static_cast<float>(beta);
    const int r_base = it.tile_r * kTile, c_base = it.tile_c * kTile;
    float xv[16];
    load_phat<TX>(md, X, r_base, c_base, tile, xv);
    const int c = c_base + threadIdx.x % kTile;
    if (c >= md.n) return;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const int r = r_base + threadIdx.x / kTile + k * kRowsPerPass;
        if (r >= md.m) continue;
        const int64_t idx = static_cast<int64_t>(r) * md.n + c;
        const float w = load_w<TW>(W, idx);
        TW* g = reinterpret_cast<TW*>(G) + idx;
        *g = from_f<TW>(to_f<TW>(*g) + (fa * xv[k] - fb * w));
    }
}

template <template <typename, typename> class K>
struct Dummy;

}  // namespace

cudaError_t launch_sumsq(const MemLaunch& p, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    if (p.wdtype == 0)
        sumsq_kernel<float><<<p.num_items, kThreads, 0, s>>>(p);
    else
        sumsq_kernel<__nv_bfloat16><<<p.num_items, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

#define SLORR_DISPATCH_WX(KERNEL)                                                         \
    do {                                                                                  \
        if (p.wdtype == 0) {                                                              \
            if (p.elem == kF32) KERNEL<float, float><<<p.num_items, kThreads, 0, s>>>(p); \
            else if (p.elem == kF16) KERNEL<float, __half><<<p.num_items, kThreads, 0, s>>>(p); \
            else KERNEL<float, __nv_bfloat16><<<p.num_items, kThreads, 0, s>>>(p);       \
        } else {                                                                          \
            if (p.elem == kF32) KERNEL<__nv_bfloat16, float><<<p.num_items, kThreads, 0, s>>>(p); \
            else if (p.elem == kF16) KERNEL<__nv_bfloat16, __half><<<p.num_items, kThreads, 0, s>>>(p); \
            else KERNEL<__nv_bfloat16, __nv_bfloat16><<<p.num_items, kThreads, 0, s>>>(p); \
        }                                                                                 \
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
