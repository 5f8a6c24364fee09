// Grouped SIMT (CUDA-core) GEMM for the three phases of a Polar Express step
// (Sec. 3 "Computational cost": A = X X^T, M = a I + b A + c A^2, X <- M X on
// the P x Q Gram side; M X is the step's a X + (b A + c A^2) X).  Used for the fp32 compute mode and, with 16-bit
// storage, as a CUDA-core check of the tensor-core kernel.  64 x 64 output
// tile per block, 256 threads, 4 x 4 per thread, K staged 16 at a time through
// shared memory.
//
// In fp32 mode the dot products are compensated (Ogita-Rump-Oishi "Dot2":
// each product is split exactly with an FMA, each addition with Knuth's
// two-sum, and the error terms are summed separately), so a result is as
// accurate as if it had been accumulated in twice the working precision and
// only the fp32 storage of X, A and B rounds.  Plain fp32 accumulation of the
// K <= 4608 long sums loses up to ~1e-5 on the Hoyer gradient of wide,
// near-full-rank matrices; the compensated sums stay near 4e-7.  The 16-bit
// check path keeps plain fp32 FMA accumulation, like the tensor cores.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "internal.h"

namespace slorr {
namespace {

constexpr int kBM = 64, kBN = 64, kBK = 16;

template <typename T>
__device__ __forceinline__ float ld_f(const T* p);
template <>
__device__ __forceinline__ float ld_f<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ld_f<__half>(const __half* p) { return __half2float(*p); }
template <>
__device__ __forceinline__ float ld_f<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }

template <typename T>
__device__ __forceinline__ void st_f(T* p, float v);
template <>
__device__ __forceinline__ void st_f<float>(float* p, float v) { *p = v; }
template <>
__device__ __forceinline__ void st_f<__half>(__half* p, float v) { *p = __float2half_rn(v); }
template <>
__device__ __forceinline__ void st_f<__nv_bfloat16>(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

template <typename T>
__global__ void __launch_bounds__(256) simt_gemm_kernel(const GemmLaunch p) {
    __shared__ float As[kBK][kBM + 4];
    __shared__ float Bs[kBK][kBN + 4];
    const GemmItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const T* X = reinterpret_cast<const T*>(md.x[p.cur]);
    const T* Am = reinterpret_cast<const T*>(md.a);
    const T* Bm = reinterpret_cast<const T*>(md.b);
    // X(p, q) lives at xb[p * sp + q * sq] (the buffer is in W's orientation).
    const int64_t sp = md.transposed ? 1 : md.ld, sq = md.transposed ? md.ld : 1;
    // Operands: Aop(i, k) = opA[i * sa_i + k * sa_k]; Bop(k, j) = opB[j * sb_j + k * sb_k].
    const T* opA;
    const T* opB;
    int64_t sa_i, sa_k, sb_j, sb_k;
    int K;
    if (p.phase == kGram) {          // A = X X^T
        opA = X; sa_i = sp; sa_k = sq; opB = X; sb_j = sp; sb_k = sq; K = md.Qpad;
    } else if (p.phase == kPoly) {   // A A
        opA = Am; sa_i = md.Ppad; sa_k = 1; opB = Am; sb_j = md.Ppad; sb_k = 1; K = md.Ppad;
    } else {                         // M X
        opA = Bm; sa_i = md.Ppad; sa_k = 1; opB = X; sb_j = sq; sb_k = sp; K = md.Ppad;
    }
    const int m0 = it.tm * kBM, n0 = it.tn * kBN;
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    constexpr bool kDot2 = sizeof(T) == 4;
    float acc[4][4] = {};
    float cmp[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += kBK) {
        // 64 x 16 of each operand: 1024 values, 4 per thread.
        for (int e = threadIdx.x; e < kBM * kBK; e += 256) {
            int i, k;
            if (sa_k == 1) { i = e / kBK; k = e % kBK; } else { k = e / kBM; i = e % kBM; }
            As[k][i] = ld_f<T>(opA + static_cast<int64_t>(m0 + i) * sa_i + static_cast<int64_t>(k0 + k) * sa_k);
        }
        for (int e = threadIdx.x; e < kBN * kBK; e += 256) {
            int j, k;
            if (sb_k == 1) { j = e / kBK; k = e % kBK; } else { k = e / kBN; j = e % kBN; }
            Bs[k][j] = ld_f<T>(opB + static_cast<int64_t>(n0 + j) * sb_j + static_cast<int64_t>(k0 + k) * sb_k);
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < kBK; ++k) {
            float a[4], b[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) a[u] = As[k][ty * 4 + u];
#pragma unroll
            for (int v = 0; v < 4; ++v) b[v] = Bs[k][tx * 4 + v];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    if constexpr (kDot2) {
                        const float pr = a[u] * b[v];
                        const float pe = fmaf(a[u], b[v], -pr);   // a b = pr + pe exactly
                        const float s = acc[u][v] + pr;
                        const float z = s - acc[u][v];
                        const float se = (acc[u][v] - (s - z)) + (pr - z);  // two-sum error
                        acc[u][v] = s;
                        cmp[u][v] += pe + se;
                    } else {
                        acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
                    }
                }
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int i = m0 + ty * 4 + u, j = n0 + tx * 4 + v;
            const float acc_uv = acc[u][v] + cmp[u][v];
            if (p.phase == kGram) {
                st_f<T>(reinterpret_cast<T*>(md.a) + static_cast<int64_t>(i) * md.Ppad + j, acc_uv);
            } else if (p.phase == kPoly) {      // M = c A^2 + b A + a I
                const int64_t idx = static_cast<int64_t>(i) * md.Ppad + j;
                float val = fmaf(p.b, ld_f<T>(Am + idx), p.c * acc_uv);
                if (i == j) val += p.a;
                st_f<T>(reinterpret_cast<T*>(md.b) + idx, val);
            } else {                            // X' = M X
                st_f<T>(reinterpret_cast<T*>(md.x[p.cur ^ 1]) + static_cast<int64_t>(i) * sp +
                            static_cast<int64_t>(j) * sq, acc_uv);
            }
        }
    }
}

}  // namespace

cudaError_t launch_gemm_simt(const GemmLaunch& p, int elem, cudaStream_t s) {
    if (p.num_items == 0) return cudaSuccess;
    if (elem == kF32)
        simt_gemm_kernel<float><<<p.num_items, 256, 0, s>>>(p);
    else if (elem == kF16)
        simt_gemm_kernel<__half><<<p.num_items, 256, 0, s>>>(p);
    else
        simt_gemm_kernel<__nv_bfloat16><<<p.num_items, 256, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace slorr
