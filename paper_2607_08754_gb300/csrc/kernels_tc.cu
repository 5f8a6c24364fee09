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

#include "internal.h"
#include "ptx.cuh"

namespace slorr {
namespace {

constexpr int kBM = 128;       // rows of one UMMA
constexpr int kBNMax = 256;
constexpr int kTmemCols = 512;
constexpr int kAccCols = 256;  // fp32 columns of one 128 x 256 accumulator
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
// or above the diagonal are computed.  Tile (tm, tn) covers row blocks from
// tm MT on and column blocks 2 tn .. min(2 tn + 1, nb - 1) (nb = Ppad / 128), so
// it is computed iff its last column block reaches its first row block.
__device__ __forceinline__ bool sym_tile_computed(int tm, int tn, int Ppad, int mt) {
    const int last_col_block = min(2 * tn + 1, Ppad / 128 - 1);
    return last_col_block >= tm * mt;
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
            const int row = row0 + quad * 32 + lane;
            const uint32_t t_row =
                tmem_base + (uint32_t(quad * 32) << 16) + uint32_t((slot + half) * kAccCols);
            const int nch = it.nsz / 32;
            if (p.phase == kUpdate) {
                uint16_t* out = reinterpret_cast<uint16_t*>(md.x[p.cur ^ 1]);
                const int64_t ld = md.ld;
                for (int ch = 0; ch < nch; ++ch) {
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
                // Poly reads b A at the output position: loads for the next chunk are
                // issued before the current chunk is processed.
                uint4 e_next[4];
                if (poly) {
                    const uint4* src = reinterpret_cast<const uint4*>(amat + int64_t(row) * ld + it.tn * kBNMax);
#pragma unroll
                    for (int q = 0; q < 4; ++q) e_next[q] = src[q];
                }
                for (int ch = 0; ch < nch; ++ch) {
                    const int col0 = it.tn * kBNMax + ch * 32;
                    const int64_t off = int64_t(row) * ld + col0;
                    uint4 e[4];
                    if (poly) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) e[q] = e_next[q];
                        if (ch + 1 < nch) {
                            const uint4* src = reinterpret_cast<const uint4*>(amat + off + 32);
#pragma unroll
                            for (int q = 0; q < 4; ++q) e_next[q] = src[q];
                        }
                    }
                    uint32_t r[32];
                    ptx::tmem_ld_32x32b_x32(t_row + uint32_t(ch * 32), r);
                    ptx::tmem_ld_wait();
                    uint4 o[4];
                    uint32_t* ow = reinterpret_cast<uint32_t*>(o);
                    const int d = row - col0;  // diagonal element of this row, if in the chunk
                    const uint32_t* ew = reinterpret_cast<const uint32_t*>(e);
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        float lo = cacc * __uint_as_float(r[2 * j]);
                        float hi = cacc * __uint_as_float(r[2 * j + 1]);
                        if (poly) {
                            // M = c A^2 + b A + a I
                            const float2 x = unpack2<BF16>(ew[j]);
                            lo = fmaf(p.b, x.x, lo) + (2 * j == d ? p.a : 0.f);
                            hi = fmaf(p.b, x.y, hi) + (2 * j + 1 == d ? p.a : 0.f);
                        }
                        ow[j] = pack2<BF16>(lo, hi);
                    }
                    uint4* dst = reinterpret_cast<uint4*>(out + off);
#pragma unroll
                    for (int q = 0; q < 4; ++q) dst[q] = o[q];
                    // The output is symmetric and strictly-lower tiles are skipped:
                    // write the transpose of this 128 x 128 block (I, J), J > I, when
                    // the tile that holds (J, I) is not computed.  The mirrored copy
                    // uses the same rounded 16-bit values, so the stored matrix is
                    // exactly symmetric.
                    const int I = row0 / kBM, J = col0 / kBM;
                    if (J > I && !sym_tile_computed(J / C::MT, I / 2, md.Ppad, C::MT)) {
                        uint16_t* tdst = out + int64_t(col0) * ld + row;
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            tdst[int64_t(2 * j) * ld] = uint16_t(ow[j] & 0xffffu);
                            tdst[int64_t(2 * j + 1) * ld] = uint16_t(ow[j] >> 16);
                        }
                    }
                }
            }
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
