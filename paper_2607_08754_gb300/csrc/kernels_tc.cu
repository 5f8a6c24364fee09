// Grouped persistent tensor-core GEMM for one phase of a Polar Express step
// (Sec. 3 "Computing the polar factor" / "Computational cost"):
//   Gram    A  = X X^T                 M = Ppad, N = Ppad, K = Qpad
//   Poly    M  = a I + b A + c A A     M = Ppad, N = Ppad, K = Ppad   (A symmetric)
//   Update  X' = M X                   M = Ppad, N = Qpad, K = Ppad
// over every matrix of the weight set in one launch; M X equals the step's
// a X + (b A + c A^2) X.  The iterate X is stored in W's orientation, so for
// m <= n it is a K-major operand of the Gram product and an MN-major one of
// the update, and the other way round for m > n; the UMMA descriptors take
// either form, so no transpose is ever materialised.  Operands are fp16 or
// bf16, accumulation fp32 in tensor memory.
//
// One CTA per SM (192 threads):
//   warp 0      TMA producer: 128 x 64 A-operand and nsz x 64 B-operand boxes
//               (128-byte swizzle) into a 4-stage shared-memory ring;
//   warp 1      allocates 512 TMEM columns; lane 0 issues tcgen05.mma
//               (M = 128, N = nsz <= 256, K = 16) into one of two 256-column
//               fp32 accumulators and commits stage releases / tile completion;
//   warps 2..5  epilogue: tcgen05.ld 32 columns at a time, add b A + a I
//               (Poly only) in fp32, round to 16 bit, store to global (the
//               update of an m > n matrix stores its tile transposed).
// Output tiles are 128 x nsz with nsz a multiple of 64, taken round-robin from
// a host-built list; accumulator double-buffering overlaps a tile's epilogue
// with the next tile's main loop.  Every wait is bounded; on a timeout the CTA
// records it in the status word, drains its in-flight copies and MMAs and
// returns.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"

namespace slorr {
namespace {

constexpr int kBM = 128;
constexpr int kBNMax = 256;
constexpr int kTmemCols = 512;
constexpr int kAccCols = 256;
constexpr int kThreads = 192;
constexpr int kEpiWarps = 4;
constexpr int kMaxStages = 16;

// Pipeline configuration: K depth of a stage and number of stages.
//   BK = 64 (default): K-major boxes are 64 x 64 with the 128-byte swizzle,
//                      48 KB stages, 4 stages;
//   BK = 32 (option):  K-major boxes are 32 x 64 with the 64-byte swizzle,
//                      24 KB stages, 9 stages.  Deeper, but its 64-byte rows
//                      halve the bytes per L2 request; measured 1.5x slower.
// MN-major boxes are always 64 (MN) x BK rows with the 128-byte swizzle.  Every
// box holds 64 x BK elements.
template <int BK_, int STAGES_>
struct Cfg {
    static constexpr int BK = BK_;
    static constexpr int STAGES = STAGES_;
    static constexpr int kBoxBytes = 64 * BK * 2;
    static constexpr int kABytes = kBM * BK * 2;
    static constexpr int kBBytes = kBNMax * BK * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr uint32_t kKLayout = BK == 64 ? 2u : 4u;  // SWIZZLE_128B / SWIZZLE_64B
    static constexpr uint32_t kKSbo = 8 * BK * 2;              // 8 rows of BK 16-bit elements
    static constexpr size_t kSmemBytes = size_t(STAGES) * kStageBytes + 1024 /*align*/ + 256 /*barriers*/;
    static_assert(STAGES <= kMaxStages, "too many stages");
    static_assert(kSmemBytes <= 232448, "shared memory budget");
};
using Cfg64 = Cfg<64, 4>;
using Cfg32 = Cfg<32, 9>;

template <bool BF16>
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    if constexpr (BF16) {
        __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        return *reinterpret_cast<uint32_t*>(&v);
    } else {
        __half2 v = __floats2half2_rn(lo, hi);
        return *reinterpret_cast<uint32_t*>(&v);
    }
}

template <bool BF16>
__device__ __forceinline__ uint16_t to16(float x) {
    if constexpr (BF16)
        return __bfloat16_as_ushort(__float2bfloat16_rn(x));
    else
        return __half_as_ushort(__float2half_rn(x));
}

template <bool BF16>
__device__ __forceinline__ float2 unpack2(uint32_t u) {
    if constexpr (BF16) {
        __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
        return __bfloat1622float2(v);
    } else {
        __half2 v = *reinterpret_cast<__half2*>(&u);
        return __half22float2(v);
    }
}

struct Smem {
    uint8_t* stages;
    uint64_t* full;
    uint64_t* empty;
    uint64_t* tfull;
    uint64_t* tempty;
    uint64_t* drain;
    uint32_t* tmem_slot;
    volatile int* abort;
    volatile int* never;  // stays 0: drain waits ignore the abort flag
};

__device__ __forceinline__ void record_timeout(const GemmLaunch& p, const Smem& s) {
    *s.abort = 1;
    atomicOr(p.status, kStatusTimeout);
}

struct PhaseInfo {
    const void* mapA;
    const void* mapB;
    int nkb;
    bool a_mn;   // A operand MN-major (else K-major)
    bool b_mn;   // B operand MN-major (else K-major)
};

// Tensor maps per matrix (kMapsPerMatrix of them, 128 bytes each):
// X0 K-major, X1 K-major, X0 MN-major, X1 MN-major, A K-major, M K-major.
__device__ __forceinline__ const void* xmap(const uint8_t* maps, int buf, bool mn) {
    return maps + (mn ? 2 + buf : buf) * 128;
}

template <class C>
__device__ __forceinline__ PhaseInfo phase_info(const GemmLaunch& p, const GemmItem& it) {
    const MatDev& md = p.mats[it.mat];
    const uint8_t* maps = reinterpret_cast<const uint8_t*>(p.maps) + size_t(it.mat) * kMapsPerMatrix * 128;
    const bool tr = md.transposed != 0;
    PhaseInfo pi;
    if (p.phase == kGram) {
        pi.a_mn = tr;
        pi.b_mn = tr;
        pi.mapA = xmap(maps, p.cur, tr);
        pi.mapB = pi.mapA;
        pi.nkb = md.Qpad / C::BK;
    } else if (p.phase == kPoly) {
        pi.a_mn = false;
        pi.b_mn = false;
        pi.mapA = maps + 4 * 128;
        pi.mapB = pi.mapA;
        pi.nkb = md.Ppad / C::BK;
    } else {
        pi.a_mn = false;
        pi.b_mn = !tr;
        pi.mapA = maps + 5 * 128;
        pi.mapB = xmap(maps, p.cur, pi.b_mn);
        pi.nkb = md.Ppad / C::BK;
    }
    return pi;
}

// Symmetric products (Gram, Poly): only tiles holding some 128 x 128 block on
// or above the diagonal are computed.  Tile (tm, tn) covers column blocks
// 2 tn .. 2 tn + nblk - 1 (nblk = nsz / 128), so it is computed iff its last
// column block reaches the diagonal: 2 tn + nblk - 1 >= tm.
__device__ __forceinline__ bool sym_tile_computed(int tm, int tn, int Ppad) {
    const int last_block = min(2 * tn + 1, Ppad / 128 - 1);
    return last_block >= tm;
}

// Shared-memory descriptor of one K = 16 slice (kk) of a BK-wide K block:
// K-major: rows of 2 BK bytes (swizzle span), 8-row groups kKSbo apart, slice
// kk starts 32 bytes further inside the swizzle atom; MN-major: 64-element MN
// chunks one box apart (LBO), 8-row K groups 1 KB apart (SBO), slice kk starts
// 16 rows = 2 KB further.
template <class C>
__device__ __forceinline__ uint64_t operand_desc(uint32_t base, int kk, bool mn) {
    return mn ? ptx::sdesc(base + kk * 16 * 128, C::kBoxBytes, 1024, 2u)
              : ptx::sdesc(base + kk * 32, 16, C::kKSbo, C::kKLayout);
}

template <class C>
__device__ void producer(const GemmLaunch& p, const Smem& s) {
    int stage = 0;
    uint32_t phase = 0;
    int issued_parity[C::STAGES];
#pragma unroll
    for (int i = 0; i < C::STAGES; ++i) issued_parity[i] = -1;
    bool ok = true;
    for (int idx = blockIdx.x; idx < p.num_items && ok; idx += gridDim.x) {
        const GemmItem it = p.items[idx];
        const PhaseInfo pi = phase_info<C>(p, it);
        const uint32_t bytes = C::kABytes + uint32_t(it.nsz) * C::BK * 2;
        const int nboxes = it.nsz / 64;
        for (int kb = 0; kb < pi.nkb; ++kb) {
            if (!ptx::mbar_wait(&s.empty[stage], phase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            uint8_t* sa = s.stages + size_t(stage) * C::kStageBytes;
            uint8_t* sb = sa + C::kABytes;
            ptx::mbar_arrive_expect_tx(&s.full[stage], bytes);
            // box coordinates are (inner, outer): (k, mn) for K-major, (mn, k) for MN-major
            for (int h = 0; h < 2; ++h) {
                const int mn = it.tm * kBM + h * 64, k = kb * C::BK;
                ptx::tma_load_2d(sa + h * C::kBoxBytes, pi.mapA, &s.full[stage], pi.a_mn ? mn : k,
                                 pi.a_mn ? k : mn);
            }
            for (int j = 0; j < nboxes; ++j) {
                const int mn = it.tn * kBNMax + j * 64, k = kb * C::BK;
                ptx::tma_load_2d(sb + j * C::kBoxBytes, pi.mapB, &s.full[stage], pi.b_mn ? mn : k,
                                 pi.b_mn ? k : mn);
            }
            if (p.prefetch > 0 && kb + p.prefetch < pi.nkb) {
                // warm L2 with the k block `prefetch` steps ahead of this one
                const int k = (kb + p.prefetch) * C::BK;
                for (int h = 0; h < 2; ++h) {
                    const int mn = it.tm * kBM + h * 64;
                    ptx::tma_prefetch_l2_2d(pi.mapA, pi.a_mn ? mn : k, pi.a_mn ? k : mn);
                }
                for (int j = 0; j < nboxes; ++j) {
                    const int mn = it.tn * kBNMax + j * 64;
                    ptx::tma_prefetch_l2_2d(pi.mapB, pi.b_mn ? mn : k, pi.b_mn ? k : mn);
                }
            }
            issued_parity[stage] = int(phase);
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
    if (!ok) {
        // Wait (bounded) for every copy this thread issued to land before exit.
        for (int i = 0; i < C::STAGES; ++i)
            if (issued_parity[i] >= 0)
                ptx::mbar_wait(&s.full[i], uint32_t(issued_parity[i]), s.never, p.timeout_ns);
    }
}

template <bool BF16, class C>
__device__ void mma_issuer(const GemmLaunch& p, const Smem& s, uint32_t tmem_base) {
    int stage = 0;
    uint32_t phase = 0;
    int local = 0;
    bool ok = true;
    bool issued_any = false;
    for (int idx = blockIdx.x; idx < p.num_items && ok; idx += gridDim.x, ++local) {
        const GemmItem it = p.items[idx];
        const PhaseInfo pi = phase_info<C>(p, it);
        const uint32_t idesc = ptx::idesc_f16(kBM, it.nsz, BF16, pi.a_mn, pi.b_mn);
        const int buf = local & 1;
        const uint32_t tphase = (uint32_t(local) >> 1) & 1u;
        if (!ptx::mbar_wait(&s.tempty[buf], tphase ^ 1u, s.abort, p.timeout_ns)) {
            record_timeout(p, s);
            ok = false;
            break;
        }
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem_base + uint32_t(buf * kAccCols);
        for (int kb = 0; kb < pi.nkb; ++kb) {
            if (!ptx::mbar_wait(&s.full[stage], phase, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            const uint32_t a0 = ptx::smem_u32(s.stages + size_t(stage) * C::kStageBytes);
            const uint32_t b0 = a0 + C::kABytes;
#pragma unroll
            for (int kk = 0; kk < C::BK / 16; ++kk) {
                ptx::umma_f16(d_tmem, operand_desc<C>(a0, kk, pi.a_mn), operand_desc<C>(b0, kk, pi.b_mn), idesc,
                              (kb | kk) != 0 ? 1u : 0u);
            }
            issued_any = true;
            ptx::umma_commit(&s.empty[stage]);
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        ptx::umma_commit(&s.tfull[buf]);
    }
    if (!ok && issued_any) {
        // Make sure no MMA is still writing TMEM before it is released.
        ptx::umma_commit(s.drain);
        ptx::mbar_wait(s.drain, 0u, s.never, p.timeout_ns);
    }
}

template <bool BF16>
__device__ void epilogue(const GemmLaunch& p, const Smem& s, uint32_t tmem_base, int warp,
                         int lane) {
    const int quad = warp & 3;  // TMEM lanes [32 quad, 32 quad + 32)
    int local = 0;
    for (int idx = blockIdx.x; idx < p.num_items; idx += gridDim.x, ++local) {
        const GemmItem it = p.items[idx];
        const MatDev& md = p.mats[it.mat];
        const int buf = local & 1;
        const uint32_t tphase = (uint32_t(local) >> 1) & 1u;
        int ok = 1;
        if (lane == 0) ok = ptx::mbar_wait(&s.tfull[buf], tphase, s.abort, p.timeout_ns) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) record_timeout(p, s);
            break;
        }
        ptx::tc_fence_after();
        const int row = it.tm * kBM + quad * 32 + lane;
        const uint32_t t_row = tmem_base + (uint32_t(quad * 32) << 16) + uint32_t(buf * kAccCols);
        if (p.phase == kUpdate) {
            uint16_t* out = reinterpret_cast<uint16_t*>(md.x[p.cur ^ 1]);
            const int64_t ld = md.ld;
            for (int ch = 0; ch < it.nsz / 32; ++ch) {
                uint32_t r[32];
                ptx::tmem_ld_32x32b_x32(t_row + uint32_t(ch * 32), r);
                ptx::tmem_ld_wait();
                const int col0 = it.tn * kBNMax + ch * 32;
                if (md.transposed) {
                    // X^T[q][p]: for each column the warp's 32 rows are contiguous
                    uint16_t* dst = out + int64_t(col0) * ld + row;
#pragma unroll
                    for (int j = 0; j < 32; ++j) dst[int64_t(j) * ld] = to16<BF16>(__uint_as_float(r[j]));
                } else {
                    uint4 o[4];
                    uint32_t* ow = reinterpret_cast<uint32_t*>(o);
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        ow[j] = pack2<BF16>(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
                    uint4* dst = reinterpret_cast<uint4*>(out + int64_t(row) * ld + col0);
#pragma unroll
                    for (int v = 0; v < 4; ++v) dst[v] = o[v];
                }
            }
        } else {
            uint16_t* out = reinterpret_cast<uint16_t*>(p.phase == kGram ? md.a : md.b);
            const uint16_t* amat = reinterpret_cast<const uint16_t*>(md.a);
            const int64_t ld = md.Ppad;
            const bool poly = p.phase == kPoly;
            const float cacc = poly ? p.c : 1.f;
            for (int ch = 0; ch < it.nsz / 32; ++ch) {
                uint32_t r[32];
                ptx::tmem_ld_32x32b_x32(t_row + uint32_t(ch * 32), r);
                ptx::tmem_ld_wait();
                const int col0 = it.tn * kBNMax + ch * 32;
                const int64_t off = int64_t(row) * ld + col0;
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = cacc * __uint_as_float(r[j]);
                if (poly) {
                    // M = c A^2 + b A + a I
                    uint4 e[4];
                    const uint4* src = reinterpret_cast<const uint4*>(amat + off);
#pragma unroll
                    for (int q = 0; q < 4; ++q) e[q] = src[q];
                    const uint32_t* ew = reinterpret_cast<const uint32_t*>(e);
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float2 x = unpack2<BF16>(ew[j]);
                        v[2 * j] = fmaf(p.b, x.x, v[2 * j]);
                        v[2 * j + 1] = fmaf(p.b, x.y, v[2 * j + 1]);
                    }
                    const int d = row - col0;
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j == d) v[j] += p.a;
                }
                uint4 o[4];
                uint32_t* ow = reinterpret_cast<uint32_t*>(o);
#pragma unroll
                for (int j = 0; j < 16; ++j) ow[j] = pack2<BF16>(v[2 * j], v[2 * j + 1]);
                uint4* dst = reinterpret_cast<uint4*>(out + off);
#pragma unroll
                for (int q = 0; q < 4; ++q) dst[q] = o[q];
                // The output is symmetric and strictly-lower tiles are skipped:
                // write the transpose of this 128 x 128 block (I, J), J > I, when
                // the tile that holds (J, I) is not computed.
                const int I = it.tm, J = col0 / 128;
                if (J > I && !sym_tile_computed(J, I / 2, md.Ppad)) {
                    uint16_t* tdst = out + int64_t(col0) * ld + row;
#pragma unroll
                    for (int j = 0; j < 32; ++j) tdst[int64_t(j) * ld] = to16<BF16>(v[j]);
                }
            }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&s.tempty[buf]);
    }
}

template <bool BF16, class C>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const __grid_constant__ GemmLaunch p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    Smem s;
    s.stages = base;
    s.full = reinterpret_cast<uint64_t*>(base + size_t(C::STAGES) * C::kStageBytes);
    s.empty = s.full + C::STAGES;
    s.tfull = s.empty + C::STAGES;
    s.tempty = s.tfull + 2;
    s.drain = s.tempty + 2;
    s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
    s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
    s.never = s.abort + 1;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::STAGES; ++i) {
            ptx::mbar_init(&s.full[i], 1);
            ptx::mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&s.tfull[i], 1);
            ptx::mbar_init(&s.tempty[i], kEpiWarps);
        }
        ptx::mbar_init(s.drain, 1);
        *s.abort = 0;
        *s.never = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        // Warm the descriptors of the first item.
        if (blockIdx.x < p.num_items) {
            const PhaseInfo pi = phase_info<C>(p, p.items[blockIdx.x]);
            ptx::prefetch_tmap(pi.mapA);
            ptx::prefetch_tmap(pi.mapB);
        }
    }
    if (warp == 1) {
        ptx::tmem_alloc(s.tmem_slot, kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *s.tmem_slot;

    if (warp == 0) {
        if (lane == 0) producer<C>(p, s);
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) mma_issuer<BF16, C>(p, s, tmem_base);
        __syncwarp();
    } else {
        epilogue<BF16>(p, s, tmem_base, warp, lane);
    }
    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, kTmemCols);
    }
}

template <bool BF16, class C>
cudaError_t launch_cfg(const GemmLaunch& p, int grid, cudaStream_t st) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(tc_gemm_kernel<BF16, C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             int(C::kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    tc_gemm_kernel<BF16, C><<<grid, kThreads, C::kSmemBytes, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_tc(const GemmLaunch& p, int elem, int grid, cudaStream_t st) {
    if (p.num_items == 0) return cudaSuccess;
    if (grid > p.num_items) grid = p.num_items;
    const bool bf = elem == kBF16;
    if (p.bk == 32) return bf ? launch_cfg<true, Cfg32>(p, grid, st) : launch_cfg<false, Cfg32>(p, grid, st);
    return bf ? launch_cfg<true, Cfg64>(p, grid, st) : launch_cfg<false, Cfg64>(p, grid, st);
}

}  // namespace slorr
