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
// One CTA per SM, warp-specialised:
//   warp 0        TMA producer: A-operand (MT x 128 rows x BK) and B-operand
//                 (nsz x BK) boxes into a STAGES-deep shared-memory ring;
//   warp 1        allocates all 512 TMEM columns; lane 0 issues tcgen05.mma
//                 (M = 128, N = nsz <= 256, K = 16), one per 128-row M tile,
//                 and commits stage releases / tile completion;
//   warps 2..     4 x MT epilogue warps: tcgen05.ld 32 columns at a time, add
//                 b A + a I (Poly only) in fp32, round to 16 bit, store (the
//                 update of an m > n matrix stores its tile transposed).
// A CTA tile is (MT x 128) x nsz.  MT = 1: two 256-column accumulators, so a
// tile's epilogue overlaps the next tile's main loop.  MT = 2: one 256 x 256
// tile fills TMEM, the B tile in shared memory feeds both M halves, so each
// stage moves a third fewer 128-byte rows per FLOP (the TMA row rate is what
// bounds the main loop), at the price of an epilogue that no longer overlaps.
// Tiles are taken round-robin from a host-built list.  Every wait is bounded;
// on a timeout the CTA records it in the status word, drains its in-flight
// copies and MMAs and returns.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "tc_common.cuh"

namespace slorr {
namespace {

using namespace tc;

constexpr int kTmemCols = 512;
constexpr int kMaxStages = 16;

// Pipeline configuration: K depth BK of a stage, stages, M tiles per CTA.
//   BK = 64: K-major boxes are 64 x 64 with the 128-byte swizzle;
//   BK = 32: K-major boxes are 32 x 64 with the 64-byte swizzle (half the bytes
//            per L2 request; measured 1.5x slower, kept as a tuning option).
// MN-major boxes are always 64 (MN) x BK rows with the 128-byte swizzle.  Every
// box holds 64 x BK elements.
template <int BK_, int STAGES_, int MT_>
struct Cfg {
    static constexpr int BK = BK_;
    static constexpr int STAGES = STAGES_;
    static constexpr int MT = MT_;
    static constexpr int kBoxBytes = 64 * BK * 2;
    static constexpr int kAHalfBytes = kBM * BK * 2;  // one 128-row M tile
    static constexpr int kABytes = MT * kAHalfBytes;
    static constexpr int kBBytes = kBNMax * BK * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kSlots = MT == 1 ? 2 : 1;    // accumulator sets in TMEM
    static constexpr int kEpiWarps = 4 * MT;
    static constexpr int kThreads = 64 + 32 * kEpiWarps;
    static constexpr uint32_t kKLayout = BK == 64 ? 2u : 4u;  // SWIZZLE_128B / SWIZZLE_64B
    static constexpr uint32_t kKSbo = 8 * BK * 2;              // 8 rows of BK 16-bit elements
    static constexpr size_t kSmemBytes = size_t(STAGES) * kStageBytes + 1024 /*align*/ + 256 /*barriers*/;
    static_assert(STAGES <= kMaxStages, "too many stages");
    static_assert(kSmemBytes <= 232448, "shared memory budget");
    static_assert(kSlots * MT * kAccCols <= kTmemCols, "tensor memory budget");
};
using Cfg64 = Cfg<64, 4, 1>;
using Cfg32 = Cfg<32, 9, 1>;
using Cfg256 = Cfg<64, 3, 2>;

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
        const int mhalves = it.msz / kBM;
        const int nboxes = it.nsz / 64;
        const uint32_t bytes = uint32_t(mhalves) * C::kAHalfBytes + uint32_t(it.nsz) * C::BK * 2;
        for (int kb = 0; kb < pi.nkb; ++kb) {
            if (!ptx::mbar_wait(&s.empty[stage], phase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            uint8_t* sa = s.stages + size_t(stage) * C::kStageBytes;
            uint8_t* sb = sa + C::kABytes;
            const int k = kb * C::BK;
            ptx::mbar_arrive_expect_tx(&s.full[stage], bytes);
            // box coordinates are (inner, outer): (k, mn) for K-major, (mn, k) for MN-major
            for (int h = 0; h < mhalves; ++h)
                for (int b = 0; b < 2; ++b) {
                    const int mn = it.tm * (kBM * C::MT) + h * kBM + b * 64;
                    ptx::tma_load_2d(sa + h * C::kAHalfBytes + b * C::kBoxBytes, pi.mapA, &s.full[stage],
                                     pi.a_mn ? mn : k, pi.a_mn ? k : mn);
                }
            for (int j = 0; j < nboxes; ++j) {
                const int mn = it.tn * kBNMax + j * 64;
                ptx::tma_load_2d(sb + j * C::kBoxBytes, pi.mapB, &s.full[stage], pi.b_mn ? mn : k,
                                 pi.b_mn ? k : mn);
            }
            if (p.prefetch > 0 && kb + p.prefetch < pi.nkb) {
                // warm L2 with the k block `prefetch` steps ahead of this one
                const int kp = (kb + p.prefetch) * C::BK;
                for (int h = 0; h < mhalves; ++h)
                    for (int b = 0; b < 2; ++b) {
                        const int mn = it.tm * (kBM * C::MT) + h * kBM + b * 64;
                        ptx::tma_prefetch_l2_2d(pi.mapA, pi.a_mn ? mn : kp, pi.a_mn ? kp : mn);
                    }
                for (int j = 0; j < nboxes; ++j) {
                    const int mn = it.tn * kBNMax + j * 64;
                    ptx::tma_prefetch_l2_2d(pi.mapB, pi.b_mn ? mn : kp, pi.b_mn ? kp : mn);
                }
            }
            issued_parity[stage] = int(phase);
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
    if (!ok || *s.abort) {
        // Some role gave up, so the MMA thread may not have consumed every stage:
        // wait (bounded) for every copy this thread issued to land before exit.
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
    if (p.test_stall) {
        // Failure-detection test: wait on the drain barrier, which nothing
        // arrives on before the end, so the bounded wait runs out and the CTA
        // takes its timeout path.
        if (!ptx::mbar_wait(s.drain, 0u, s.abort, p.timeout_ns)) {
            record_timeout(p, s);
            ok = false;
        }
    }
    for (int idx = blockIdx.x; idx < p.num_items && ok; idx += gridDim.x, ++local) {
        const GemmItem it = p.items[idx];
        const PhaseInfo pi = phase_info<C>(p, it);
        const uint32_t idesc = ptx::idesc_f16(kBM, it.nsz, BF16, pi.a_mn, pi.b_mn);
        const int mhalves = it.msz / kBM;
        const int slot = local % C::kSlots;
        const uint32_t tphase = uint32_t(local / C::kSlots) & 1u;
        if (!ptx::mbar_wait(&s.tempty[slot], tphase ^ 1u, s.abort, p.timeout_ns)) {
            record_timeout(p, s);
            ok = false;
            break;
        }
        ptx::tc_fence_after();
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
                const uint64_t bd = operand_desc<C>(b0, kk, pi.b_mn);
#pragma unroll
                for (int h = 0; h < C::MT; ++h) {
                    if (h < mhalves) {
                        const uint32_t d_tmem = tmem_base + uint32_t((slot + h) * kAccCols);
                        ptx::umma_f16(d_tmem, operand_desc<C>(a0 + h * C::kAHalfBytes, kk, pi.a_mn), bd, idesc,
                                      (kb | kk) != 0 ? 1u : 0u);
                    }
                }
            }
            issued_any = true;
            ptx::umma_commit(&s.empty[stage]);
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        ptx::umma_commit(&s.tfull[slot]);
    }
    if (!ok && issued_any) {
        // Make sure no MMA is still writing TMEM before it is released.
        ptx::umma_commit(s.drain);
        ptx::mbar_wait(s.drain, 0u, s.never, p.timeout_ns);
    }
}

template <bool BF16, class C>
__device__ void epilogue(const GemmLaunch& p, const Smem& s, uint32_t tmem_base, int warp, int lane) {
    const int quad = warp & 3;           // TMEM lanes [32 quad, 32 quad + 32) (hardware rule)
    const int half = (warp - 2) / 4;     // which 128-row M tile of the CTA tile
    int local = 0;
    for (int idx = blockIdx.x; idx < p.num_items; idx += gridDim.x, ++local) {
        const GemmItem it = p.items[idx];
        const MatDev& md = p.mats[it.mat];
        const int slot = local % C::kSlots;
        const uint32_t tphase = uint32_t(local / C::kSlots) & 1u;
        int ok = 1;
        if (lane == 0) ok = ptx::mbar_wait(&s.tfull[slot], tphase, s.abort, p.timeout_ns) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) record_timeout(p, s);
            break;
        }
        ptx::tc_fence_after();
        if (half < it.msz / kBM) {
            const int row0 = it.tm * (kBM * C::MT) + half * kBM;  // first row of this 128-row tile
            const uint32_t t_row =
                tmem_base + (uint32_t(quad * 32) << 16) + uint32_t((slot + half) * kAccCols);
            store_rows<BF16, C::MT>(p, it, md, row0, t_row, quad, lane, 0, it.nsz / 32);
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&s.tempty[slot]);
    }
}

template <bool BF16, class C>
__global__ void __launch_bounds__(C::kThreads, 1) tc_gemm_kernel(const __grid_constant__ GemmLaunch p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    Smem s;
    s.stages = base;
    s.full = reinterpret_cast<uint64_t*>(base + size_t(C::STAGES) * C::kStageBytes);
    s.empty = s.full + C::STAGES;
    s.tfull = s.empty + C::STAGES;
    s.tempty = s.tfull + C::kSlots;
    s.drain = s.tempty + C::kSlots;
    s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
    s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
    s.never = s.abort + 1;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::STAGES; ++i) {
            ptx::mbar_init(&s.full[i], 1);
            ptx::mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < C::kSlots; ++i) {
            ptx::mbar_init(&s.tfull[i], 1);
            ptx::mbar_init(&s.tempty[i], C::kEpiWarps);
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
        epilogue<BF16, C>(p, s, tmem_base, warp, lane);
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
    tc_gemm_kernel<BF16, C><<<grid, C::kThreads, C::kSmemBytes, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_tc(const GemmLaunch& p, int elem, int grid, cudaStream_t st) {
    if (p.num_items == 0) return cudaSuccess;
    if (grid > p.num_items) grid = p.num_items;
    const bool bf = elem == kBF16;
    if (p.mt == 2) return bf ? launch_cfg<true, Cfg256>(p, grid, st) : launch_cfg<false, Cfg256>(p, grid, st);
    if (p.bk == 32) return bf ? launch_cfg<true, Cfg32>(p, grid, st) : launch_cfg<false, Cfg32>(p, grid, st);
    return bf ? launch_cfg<true, Cfg64>(p, grid, st) : launch_cfg<false, Cfg64>(p, grid, st);
}

}  // namespace slorr
