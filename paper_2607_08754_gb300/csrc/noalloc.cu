// Squared Frobenius norm of one matrix with no device allocation at all.
//
// Every other entry point of libslorr needs a caller-provided workspace.  Some
// callers cannot provide one: code that runs while a CUDA stream is being
// captured (allocation is not a capturable operation), runtimes whose device
// memory is owned by a framework allocator that third-party code may not
// touch, and latency-critical loops that must never enter an allocator.  For
// them, slorr_frob_sq_noalloc() computes ||W||_F^2 -- the first quantity of the
// regularizer -- using scratch memory that is part of the library image: a
// file-scope __device__ array every GPU that loads the library holds until the
// process exits.
//
// Scratch: kMaxChunks per-chunk partial sums (256 KB).  A chunk is 8192
// elements, so one call accepts up to kMaxChunks * 8192 = 536,870,912
// elements; larger matrices are rejected.  Every partial a call reads is
// written earlier in the same call, so nothing has to start at zero, but all
// calls share the one array: calls that overlap on the GPU (other streams, or
// other host threads) race on it and must be serialised by the caller.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "../../include/slorr.h"
#include "internal.h"

namespace {

constexpr int kChunk = 8192;          // elements per block
constexpr int kThreads = 256;         // 32 elements per thread
constexpr int kMaxChunks = 65536;     // 256 KB of float partials
constexpr int kMaxDevices = 64;

static __device__ __align__(256) float g_noalloc_partials[kMaxChunks];

__device__ __forceinline__ float warp_sum(float v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// One block per chunk of the flattened matrix; writes the chunk's sum of squares.
template <typename T>
__global__ void __launch_bounds__(kThreads) noalloc_chunk_kernel(const T* __restrict__ w, int64_t count,
                                                                 float* __restrict__ partials) {
    __shared__ float red[kThreads / 32];
    const int64_t base = int64_t(blockIdx.x) * kChunk;
    float acc = 0.f;
#pragma unroll 8
    for (int i = threadIdx.x; i < kChunk; i += kThreads) {
        const int64_t idx = base + i;
        if (idx < count) {
            float v;
            if constexpr (sizeof(T) == 4)
                v = w[idx];
            else
                v = __bfloat162float(w[idx]);
            acc = fmaf(v, v, acc);
        }
    }
    acc = warp_sum(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x < 32) {
        float s = threadIdx.x < kThreads / 32 ? red[threadIdx.x] : 0.f;
        s = warp_sum(s);
        if (threadIdx.x == 0) partials[blockIdx.x] = s;
    }
}

// Adds the partials in index order (double) and writes the result.
__global__ void __launch_bounds__(kThreads) noalloc_sum_kernel(const float* __restrict__ partials, int n,
                                                               double* __restrict__ out) {
    __shared__ double red[kThreads / 32];
    double s = 0.0;
    for (int i = threadIdx.x; i < n; i += kThreads) s += double(partials[i]);
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int k = 0; k < kThreads / 32; ++k) t += red[k];
        *out = t;
    }
}

// Device address of g_noalloc_partials for each device, looked up once with
// that device current.  The array's name in host code is only a stand-in; a
// kernel must be given the address cudaGetSymbolAddress() returns.
std::mutex g_mutex;
float* g_scratch[kMaxDevices] = {};

slorr_status scratch_for_current_device(float** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        slorr::set_last_error(std::string("cudaGetDevice: ") + cudaGetErrorString(e));
        return SLORR_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) {
        slorr::set_last_error("device ordinal out of range for the no-allocation scratch table");
        return SLORR_ERR_UNSUPPORTED;
    }
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_partials);
        if (e != cudaSuccess || !p) {
            slorr::set_last_error(std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
            return e == cudaErrorNoKernelImageForDevice ? SLORR_ERR_UNSUPPORTED : SLORR_ERR_CUDA;
        }
        g_scratch[dev] = static_cast<float*>(p);
    }
    *out = g_scratch[dev];
    return SLORR_OK;
}

}  // namespace

extern "C" {

SLORR_API slorr_status slorr_frob_sq_noalloc(const void* weight, int64_t m, int64_t n, int32_t dtype,
                                             double* out_frob_sq, void* stream) {
    if (!weight || !out_frob_sq) {
        slorr::set_last_error("weight and out_frob_sq must be device pointers");
        return SLORR_ERR_INVALID_ARG;
    }
    if (m < 1 || n < 1) {
        slorr::set_last_error("matrix dimensions must be positive");
        return SLORR_ERR_INVALID_ARG;
    }
    if (dtype != SLORR_F32 && dtype != SLORR_BF16) {
        slorr::set_last_error("dtype must be SLORR_F32 or SLORR_BF16");
        return SLORR_ERR_INVALID_ARG;
    }
    if (m > (int64_t(kMaxChunks) * kChunk) / n) {
        slorr::set_last_error("matrix too large for slorr_frob_sq_noalloc: at most 536870912 elements "
                "(65536 chunks of 8192) fit its fixed scratch");
        return SLORR_ERR_INVALID_ARG;
    }
    const int64_t count = m * n;
    const int chunks = int((count + kChunk - 1) / kChunk);
    float* scratch = nullptr;
    slorr_status s = scratch_for_current_device(&scratch);
    if (s != SLORR_OK) return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (dtype == SLORR_F32)
        noalloc_chunk_kernel<float><<<chunks, kThreads, 0, st>>>(static_cast<const float*>(weight), count, scratch);
    else
        noalloc_chunk_kernel<__nv_bfloat16>
            <<<chunks, kThreads, 0, st>>>(static_cast<const __nv_bfloat16*>(weight), count, scratch);
    noalloc_sum_kernel<<<1, kThreads, 0, st>>>(scratch, chunks, out_frob_sq);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        slorr::set_last_error(std::string("launch: ") + cudaGetErrorString(e));
        return e == cudaErrorNoKernelImageForDevice ? SLORR_ERR_UNSUPPORTED : SLORR_ERR_CUDA;
    }
    return SLORR_OK;
}

}  // extern "C"
