// Grouped SIMT (CUDA-core) GEMM for the three phases of a Polar Express step
// (Sec. 3 "Computational cost": A = X X^T, M = a I + b A + c A^2, X <- M X on
// the P x Q Gram side; M X is the step's a X + (b A + c A^2) X).  Used for the
// fp32 compute mode and, with 16-bit storage, as a CUDA-core check of the
// tensor-core kernel.  32 x 32 output tile per block (small sets still fill
// the GPU), 256 threads, 2 x 2 outputs per thread, K staged 32 at a time
// through two shared-memory buffers: the next stage's global loads are in
// flight while the current one is used.  Gram and Poly are symmetric: only
// tiles on or above the diagonal are computed, and each writes its
// transposed block as well.
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

constexpr int kT = kSimtTile, kBK = 32;

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
    __shared__ float As[2][kBK][kT + 1];  // [buffer][k][i]
    __shared__ float Bs[2][kBK][kT + 1];  // [buffer][k][j]
    const GemmItem it = p.items[blockIdx.x];
    const MatDev md = p.mats[it.mat];
    const int ph = it.phase, cur = p.step & 1;  // one launch per phase and step
    const float ca = p.coef[3 * p.step], cb = p.coef[3 * p.step + 1], cc = p.coef[3 * p.step + 2];
    const T* X = reinterpret_cast<const T*>(md.x[cur]);
    const T* Am = reinterpret_cast<const T*>(md.a);
    const T* Bm = reinterpret_cast<const T*>(md.b);
    // X(p, q) lives at xb[p * sp + q * sq] (the buffer is in W's orientation).
    const int64_t sp = md.transposed ? 1 : md.ld, sq = md.transposed ? md.ld : 1;
    // Operands: Aop(i, k) = opA[i * sa_i + k * sa_k]; Bop(k, j) = opB[j * sb_j + k * sb_k].
    const T* opA;
    const T* opB;
    int64_t sa_i, sa_k, sb_j, sb_k;
    int K;
    if (ph == kGram) {               // A = X X^T
        opA = X; sa_i = sp; sa_k = sq; opB = X; sb_j = sp; sb_k = sq; K = md.Qpad;
    } else if (ph == kPoly) {        // A A
        opA = Am; sa_i = md.Ppad; sa_k = 1; opB = Am; sb_j = md.Ppad; sb_k = 1; K = md.Ppad;
    } else {                         // M X
        opA = Bm; sa_i = md.Ppad; sa_k = 1; opB = X; sb_j = sq; sb_k = sp; K = md.Ppad;
    }
    const int m0 = it.tm * kT, n0 = it.tn * kT;
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    constexpr bool kDot2 = sizeof(T) == 4;
    // Each stage: 32 x 32 values of each operand, 4 per thread, consecutive
    // threads along the operand's contiguous dimension.
    float ra[4], rb[4];
    auto gload = [&](int k0) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int e = int(threadIdx.x) + 256 * r;
            const int ia = sa_k == 1 ? e / kBK : e % kT, ka = sa_k == 1 ? e % kBK : e / kT;
            const int jb = sb_k == 1 ? e / kBK : e % kT, kb = sb_k == 1 ? e % kBK : e / kT;
            ra[r] = ld_f<T>(opA + int64_t(m0 + ia) * sa_i + int64_t(k0 + ka) * sa_k);
            rb[r] = ld_f<T>(opB + int64_t(n0 + jb) * sb_j + int64_t(k0 + kb) * sb_k);
        }
    };
    auto sstore = [&](int buf) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int e = int(threadIdx.x) + 256 * r;
            const int ia = sa_k == 1 ? e / kBK : e % kT, ka = sa_k == 1 ? e % kBK : e / kT;
            const int jb = sb_k == 1 ? e / kBK : e % kT, kb = sb_k == 1 ? e % kBK : e / kT;
            As[buf][ka][ia] = ra[r];
            Bs[buf][kb][jb] = rb[r];
        }
    };
    float acc[2][2] = {};
    float cmp[2][2] = {};
    gload(0);
    sstore(0);
    __syncthreads();
    int buf = 0;
    for (int k0 = 0; k0 < K; k0 += kBK) {
        const bool more = k0 + kBK < K;
        if (more) gload(k0 + kBK);  // in flight while this stage is used
#pragma unroll 8
        for (int k = 0; k < kBK; ++k) {
            const float a[2] = {As[buf][k][ty * 2], As[buf][k][ty * 2 + 1]};
            const float b[2] = {Bs[buf][k][tx * 2], Bs[buf][k][tx * 2 + 1]};
#pragma unroll
            for (int u = 0; u < 2; ++u)
#pragma unroll
                for (int v = 0; v < 2; ++v) {
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
        if (more) sstore(buf ^ 1);  // the other buffer: last read before the previous barrier
        __syncthreads();
        buf ^= 1;
    }
    const bool mirror = ph != kUpdate && it.tn > it.tm;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
#pragma unroll
        for (int v = 0; v < 2; ++v) {
            const int i = m0 + ty * 2 + u, j = n0 + tx * 2 + v;
            const float acc_uv = acc[u][v] + cmp[u][v];
            if (ph == kGram) {
                T* a = reinterpret_cast<T*>(md.a);
                st_f<T>(a + static_cast<int64_t>(i) * md.Ppad + j, acc_uv);
                if (mirror) st_f<T>(a + static_cast<int64_t>(j) * md.Ppad + i, acc_uv);
            } else if (ph == kPoly) {           // M = c A^2 + b A + a I (A is stored symmetric)
                const int64_t idx = static_cast<int64_t>(i) * md.Ppad + j;
                float val = fmaf(cb, ld_f<T>(Am + idx), cc * acc_uv);
                if (i == j) val += ca;
                T* m = reinterpret_cast<T*>(md.b);
                st_f<T>(m + idx, val);
                if (mirror) st_f<T>(m + static_cast<int64_t>(j) * md.Ppad + i, val);
            } else {                            // X' = M X
                st_f<T>(reinterpret_cast<T*>(md.x[cur ^ 1]) + static_cast<int64_t>(i) * sp +
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
