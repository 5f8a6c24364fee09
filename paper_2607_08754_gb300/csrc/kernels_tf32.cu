// fp32 mode on the tensor cores: the three phases of a Polar Express step
// (Sec. 3 "Computing the polar factor": Gram A = X X^T, Poly M = a I + b A +
// c A A, Update X' = M X) with fp32 operands, as three tf32 products per
// fp32 product.
//
// Every operand v is kept as hi = tf32(v) and lo = tf32(v - hi), both rounded
// to nearest, so v = hi + lo to about 2^-22 |v|.  A product x y is formed as
// hi_x hi_y + hi_x lo_y + lo_x hi_y: each term is exact in fp32 (two 11-bit
// significands), the dropped lo_x lo_y and the rounding of lo are below
// 2^-21 |x y|, and the errors are unbiased.
//
// The tensor core adds each UMMA's products into the fp32 accumulator with
// truncation, so every UMMA on an accumulator leaves a biased error of up to
// one unit of its last place: over a long K that bias, not the products,
// dominates (measured: 24 UMMAs per accumulator left 1.4e-5 on an iterate
// where the compensated CUDA-core sums leave 2e-6).  So the hi x hi products
// and the two cross products go to separate accumulators (the cross terms
// are 2^-10 smaller, so their truncation is negligible), and the MMA
// accumulates only one K block (32, four hi x hi UMMAs) into a TMEM slot; the
// epilogue adds the blocks' partial sums in registers with compensated
// (Kahan) fp32 sums while the next block accumulates in the other slot.
//
// All operands are K-major (no transposed tf32 operand forms are used): the
// Gram reads X in the Gram orientation (P x Q), the Update reads M and X^T
// (Q x P), and the Update's epilogue writes the new iterate in both
// orientations (hi and lo) and, as fp32, in W's orientation for the memory
// passes.  One CTA per 128 x 64 output tile; the symmetric Gram and Poly
// products compute only tiles that reach the diagonal, store the elements on
// and above it and mirror those above it.
//
// Roles (192 threads): warp 0 lane 0 loads the stages by TMA, warp 1
// allocates TMEM and its lane 0 issues the UMMAs, warps 2..5 are the
// epilogue (one TMEM lane quadrant each, one output row per lane).  Every
// wait is bounded; a CTA that gives up records the timeout, drains its
// UMMAs and copies and returns.
#include <atomic>
#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace slorr {
namespace {

constexpr int kTM = 128;                          // tile rows (UMMA M)
constexpr int kTN = 64;                           // tile columns (UMMA N)
constexpr int kBK = 32;                           // K per stage: 128 bytes of fp32 per row
constexpr int kStages = 4;
constexpr int kChunkBlocks = 1;                   // K blocks per TMEM accumulation chunk
constexpr int kBoxBytes = 64 * kBK * 4;           // one 64-row box, 8 KB
constexpr int kAHalf = kTM * kBK * 4;             // 128 rows of hi or lo, 16 KB
constexpr int kBHalf = kTN * kBK * 4;             // 64 rows of hi or lo, 8 KB
constexpr int kStageBytes = 2 * kAHalf + 2 * kBHalf;
constexpr int kSlots = 2;
constexpr int kSlotCols = 2 * kTN;                // per slot: hi x hi, then the cross products
constexpr uint32_t kTmemCols = 256;               // two slots
constexpr int kEpiWarps = 4;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr size_t kBarrierBytes = 256;
constexpr size_t kSmemBytes = size_t(kStages) * kStageBytes + 1024 /*align*/ + kBarrierBytes;
static_assert((2 * kStages + 2 * kSlots + 1) * 8 + 16 <= kBarrierBytes, "barrier area");
static_assert(kSmemBytes <= 232448, "shared memory budget");

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

// Operand maps of one item: A rows (the output's rows) and B rows (its
// columns), hi and lo, and the number of K blocks.
struct Ops {
    const void* a[2];
    const void* b[2];
    int nkb;
};

template <int PH>
__device__ __forceinline__ Ops item_ops(const GemmLaunch& p, const GemmItem& it) {
    const MatDev& md = p.mats[it.mat];
    const uint8_t* maps =
        reinterpret_cast<const uint8_t*>(p.tf32_maps) + size_t(it.mat) * kTf32MapsPerMatrix * 128;
    const int cur = p.step & 1;
    Ops o;
    for (int h = 0; h < 2; ++h) {
        if constexpr (PH == kGram) {
            o.a[h] = maps + (2 * cur + h) * 128;
            o.b[h] = o.a[h];
        } else if constexpr (PH == kPoly) {
            o.a[h] = maps + (8 + h) * 128;
            o.b[h] = o.a[h];
        } else {
            o.a[h] = maps + (10 + h) * 128;
            o.b[h] = maps + (4 + 2 * cur + h) * 128;
        }
    }
    o.nkb = (PH == kGram ? md.Qpad : md.Ppad) / kBK;
    return o;
}

// K-major, 128-byte swizzle: rows of 32 fp32 (one swizzle atom wide), 8-row
// groups 1 KB apart; the K = 8 slice kk starts 32 bytes further in.
__device__ __forceinline__ uint64_t kdesc(uint32_t base, int kk) { return ptx::sdesc(base + kk * 32, 16, 1024, 2u); }

template <int PH>
__device__ void producer(const GemmLaunch& p, const Smem& s) {
    int stage = 0;
    uint32_t phase = 0;
    int issued_parity[kStages];
#pragma unroll
    for (int i = 0; i < kStages; ++i) issued_parity[i] = -1;
    bool ok = true;
    for (int idx = blockIdx.x; idx < p.num_items && ok; idx += gridDim.x) {
        const GemmItem it = p.items[idx];
        const Ops o = item_ops<PH>(p, it);
        for (int kb = 0; kb < o.nkb; ++kb) {
            if (!ptx::mbar_wait(&s.empty[stage], phase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            uint8_t* st = s.stages + size_t(stage) * kStageBytes;
            const int k = kb * kBK;
            ptx::mbar_arrive_expect_tx(&s.full[stage], uint32_t(kStageBytes));
            // box coordinates are (k, row); A: two 64-row boxes per half, B: one
            for (int h = 0; h < 2; ++h) {
                for (int b = 0; b < 2; ++b)
                    ptx::tma_load_2d(st + h * kAHalf + b * kBoxBytes, o.a[h], &s.full[stage], k,
                                     it.tm * kTM + b * 64);
                ptx::tma_load_2d(st + 2 * kAHalf + h * kBHalf, o.b[h], &s.full[stage], k, it.tn * kTN);
            }
            issued_parity[stage] = int(phase);
            if (++stage == kStages) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
    if (!ok || *s.abort) {
        // Another role may have given up before consuming every stage: wait
        // (bounded) for every copy this thread issued to land before exit.
        for (int i = 0; i < kStages; ++i)
            if (issued_parity[i] >= 0) ptx::mbar_wait(&s.full[i], uint32_t(issued_parity[i]), s.never, p.timeout_ns);
    }
}

template <int PH>
__device__ void mma_issuer(const GemmLaunch& p, const Smem& s, uint32_t tmem_base) {
    constexpr uint32_t idesc = ptx::idesc_tf32(kTM, kTN);
    int stage = 0;
    uint32_t phase = 0;
    int chunk = 0;  // chunks issued so far: slot chunk % 2
    bool ok = true;
    bool issued_any = false;
    if (p.test_stall) {
        // Failure-detection test: the drain barrier gets no arrival before the
        // end, so this bounded wait runs out.
        if (!ptx::mbar_wait(s.drain, 0u, s.abort, p.timeout_ns)) {
            record_timeout(p, s);
            ok = false;
        }
    }
    for (int idx = blockIdx.x; idx < p.num_items && ok; idx += gridDim.x) {
        const GemmItem it = p.items[idx];
        const Ops o = item_ops<PH>(p, it);
        for (int kb0 = 0; kb0 < o.nkb && ok; kb0 += kChunkBlocks, ++chunk) {
            const int slot = chunk % kSlots;
            const uint32_t tphase = uint32_t(chunk / kSlots) & 1u;
            if (!ptx::mbar_wait(&s.tempty[slot], tphase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            const uint32_t d_hh = tmem_base + uint32_t(slot * kSlotCols);
            const uint32_t d_x = d_hh + uint32_t(kTN);
            const int kb1 = kb0 + kChunkBlocks < o.nkb ? kb0 + kChunkBlocks : o.nkb;
            for (int kb = kb0; kb < kb1; ++kb) {
                if (!ptx::mbar_wait(&s.full[stage], phase, s.abort, p.timeout_ns)) {
                    record_timeout(p, s);
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t st = ptx::smem_u32(s.stages + size_t(stage) * kStageBytes);
                const uint32_t ahi = st, alo = st + kAHalf, bhi = st + 2 * kAHalf, blo = bhi + kBHalf;
#pragma unroll
                for (int kk = 0; kk < kBK / 8; ++kk) {
                    const uint32_t acc = (kb != kb0 || kk != 0) ? 1u : 0u;
                    ptx::umma_tf32(d_hh, kdesc(ahi, kk), kdesc(bhi, kk), idesc, acc);
                    ptx::umma_tf32(d_x, kdesc(ahi, kk), kdesc(blo, kk), idesc, acc);
                    ptx::umma_tf32(d_x, kdesc(alo, kk), kdesc(bhi, kk), idesc, 1u);
                }
                issued_any = true;
                ptx::umma_commit(&s.empty[stage]);
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            ptx::umma_commit(&s.tfull[slot]);
        }
    }
    if (!ok && issued_any) {
        // No UMMA may still be writing TMEM when it is released.
        ptx::umma_commit(s.drain);
        ptx::mbar_wait(s.drain, 0u, s.never, p.timeout_ns);
    }
}

__device__ __forceinline__ void split_store(float v, float* hi, float* lo, int64_t off) {
    const float h = ptx::cvt_rna_tf32(v);
    hi[off] = h;
    lo[off] = ptx::cvt_rna_tf32(v - h);
}

template <int PH>
__device__ void epilogue(const GemmLaunch& p, const Smem& s, uint32_t tmem_base, int warp, int lane) {
    const int quad = warp & 3;  // TMEM lanes [32 quad, 32 quad + 32) (hardware rule)
    int chunk = 0;
    for (int idx = blockIdx.x; idx < p.num_items; idx += gridDim.x) {
        const GemmItem it = p.items[idx];
        const MatDev& md = p.mats[it.mat];
        const Ops o = item_ops<PH>(p, it);
        float sum[kTN], cmp[kTN];
#pragma unroll
        for (int j = 0; j < kTN; ++j) sum[j] = cmp[j] = 0.f;
        int ok = 1;
        for (int kb0 = 0; kb0 < o.nkb; kb0 += kChunkBlocks, ++chunk) {
            const int slot = chunk % kSlots;
            const uint32_t tphase = uint32_t(chunk / kSlots) & 1u;
            if (lane == 0) ok = ptx::mbar_wait(&s.tfull[slot], tphase, s.abort, p.timeout_ns) ? 1 : 0;
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            ptx::tc_fence_after();
            const uint32_t t_row = tmem_base + (uint32_t(quad * 32) << 16) + uint32_t(slot * kSlotCols);
#pragma unroll
            for (int half = 0; half < kTN / 32; ++half) {
                uint32_t r[32], x[32];
                ptx::tmem_ld_32x32b_x32(t_row + uint32_t(half * 32), r);
                ptx::tmem_ld_32x32b_x32(t_row + uint32_t(kTN + half * 32), x);
                ptx::tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 32; ++j) {  // compensated sum of the chunks' partials
                    const float part = __uint_as_float(r[j]) + __uint_as_float(x[j]);
                    const float y = part - cmp[half * 32 + j];
                    const float t = sum[half * 32 + j] + y;
                    cmp[half * 32 + j] = (t - sum[half * 32 + j]) - y;
                    sum[half * 32 + j] = t;
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&s.tempty[slot]);
        }
        if (!ok) {
            if (lane == 0) record_timeout(p, s);
            break;
        }
        const int i = it.tm * kTM + quad * 32 + lane;  // this lane's output row
        const int j0 = it.tn * kTN;
        const int t = p.step;
        if constexpr (PH == kUpdate) {
            const int nxt = (t & 1) ^ 1;
            const MatTf32& mt = p.tf32[it.mat];
            float* xw = reinterpret_cast<float*>(md.x[nxt]);
            float* gh = reinterpret_cast<float*>(mt.xg[nxt][0]);
            float* gl = reinterpret_cast<float*>(mt.xg[nxt][1]);
            float* uh = reinterpret_cast<float*>(mt.xu[nxt][0]);
            float* ul = reinterpret_cast<float*>(mt.xu[nxt][1]);
            const bool tr = md.transposed != 0;
#pragma unroll
            for (int jj = 0; jj < kTN; ++jj) {
                const int j = j0 + jj;
                const float v = sum[jj] + cmp[jj];
                xw[tr ? int64_t(j) * md.ld + i : int64_t(i) * md.ld + j] = v;  // W's orientation
                split_store(v, gh, gl, int64_t(i) * md.Qpad + j);
                split_store(v, uh, ul, int64_t(j) * md.Ppad + i);
            }
        } else {
            const MatTf32& mt = p.tf32[it.mat];
            const int64_t ld = md.Ppad;
            float* oh = reinterpret_cast<float*>(PH == kGram ? mt.a[0] : mt.m[0]);
            float* ol = reinterpret_cast<float*>(PH == kGram ? mt.a[1] : mt.m[1]);
            const float* ah = reinterpret_cast<const float*>(mt.a[0]);
            const float* al = reinterpret_cast<const float*>(mt.a[1]);
            const float ca = p.coef[3 * t], cb = p.coef[3 * t + 1], cc = p.coef[3 * t + 2];
#pragma unroll
            for (int jj = 0; jj < kTN; ++jj) {
                const int j = j0 + jj;
                if (j < i) continue;  // the mirror of (j, i) stores it
                float v = sum[jj] + cmp[jj];
                if constexpr (PH == kPoly) {
                    // M = c A^2 + b A + a I, with A = hi + lo
                    const int64_t e = int64_t(i) * ld + j;
                    v = fmaf(cb, __ldcg(ah + e) + __ldcg(al + e), cc * v) + (i == j ? ca : 0.f);
                }
                split_store(v, oh, ol, int64_t(i) * ld + j);
                if (j > i) split_store(v, oh, ol, int64_t(j) * ld + i);
            }
        }
    }
}

template <int PH>
__global__ void __launch_bounds__(kThreads, 1) tf32_gemm_kernel(const __grid_constant__ GemmLaunch p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    Smem s;
    s.stages = base;
    s.full = reinterpret_cast<uint64_t*>(base + size_t(kStages) * kStageBytes);
    s.empty = s.full + kStages;
    s.tfull = s.empty + kStages;
    s.tempty = s.tfull + kSlots;
    s.drain = s.tempty + kSlots;
    s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
    s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
    s.never = s.abort + 1;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            ptx::mbar_init(&s.full[i], 1);
            ptx::mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < kSlots; ++i) {
            ptx::mbar_init(&s.tfull[i], 1);
            ptx::mbar_init(&s.tempty[i], kEpiWarps);
        }
        ptx::mbar_init(s.drain, 1);
        *s.abort = 0;
        *s.never = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 0 && lane == 0 && blockIdx.x < p.num_items) {
        const Ops o = item_ops<PH>(p, p.items[blockIdx.x]);
        for (int h = 0; h < 2; ++h) {
            ptx::prefetch_tmap(o.a[h]);
            ptx::prefetch_tmap(o.b[h]);
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
    // everything above may overlap the previous kernel under programmatic
    // dependent launch; its results are read only after this
    ptx::griddep_wait();
    ptx::griddep_launch_dependents();
    if (warp == 0) {
        if (lane == 0) producer<PH>(p, s);
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) mma_issuer<PH>(p, s, tmem_base);
        __syncwarp();
    } else {
        epilogue<PH>(p, s, tmem_base, warp, lane);
    }
    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem_base, kTmemCols);
    }
}

template <int PH>
cudaError_t launch_phase(const GemmLaunch& p, cudaStream_t st) {
    static std::atomic<int> attr_done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!attr_done[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(tf32_gemm_kernel<PH>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_done[dev].store(1, std::memory_order_release);
    }
    return launch_kernel(tf32_gemm_kernel<PH>, unsigned(p.num_items), kThreads, kSmemBytes, st, p.pdl != 0, p);
}

// X_0 -> hi/lo in both orientations, one 32 x 32 tile of the Gram-orientation
// X per block (blockIdx.y: matrix), transposed through shared memory so both
// stores are coalesced.
__global__ void __launch_bounds__(256) tf32_split_kernel(const MatDev* mats, const MatTf32* tf32) {
    __shared__ float tile[32][33];
    const MatDev& md = mats[blockIdx.y];
    const int tp = md.Ppad / 32, tq = md.Qpad / 32;
    if (int(blockIdx.x) >= tp * tq) return;
    const int p0 = (int(blockIdx.x) / tq) * 32, q0 = (int(blockIdx.x) % tq) * 32;
    const float* x = reinterpret_cast<const float*>(md.x[0]);
    const int c = threadIdx.x % 32, r0 = threadIdx.x / 32;
    ptx::griddep_wait();
    for (int r = r0; r < 32; r += 8) {
        if (md.transposed)
            tile[c][r] = x[int64_t(q0 + r) * md.ld + p0 + c];  // x holds X^T: X(p0 + c, q0 + r)
        else
            tile[r][c] = x[int64_t(p0 + r) * md.ld + q0 + c];
    }
    __syncthreads();
    const MatTf32& mt = tf32[blockIdx.y];
    float* gh = reinterpret_cast<float*>(mt.xg[0][0]);
    float* gl = reinterpret_cast<float*>(mt.xg[0][1]);
    float* uh = reinterpret_cast<float*>(mt.xu[0][0]);
    float* ul = reinterpret_cast<float*>(mt.xu[0][1]);
    for (int r = r0; r < 32; r += 8) {
        split_store(tile[r][c], gh, gl, int64_t(p0 + r) * md.Qpad + q0 + c);  // X(p0 + r, q0 + c)
        split_store(tile[c][r], uh, ul, int64_t(q0 + r) * md.Ppad + p0 + c);  // X^T(q0 + r, p0 + c)
    }
    ptx::griddep_launch_dependents();
}

}  // namespace

cudaError_t launch_gemm_tf32(const GemmLaunch& p, int phase, cudaStream_t st) {
    if (p.num_items == 0) return cudaSuccess;
    switch (phase) {
        case kGram: return launch_phase<kGram>(p, st);
        case kPoly: return launch_phase<kPoly>(p, st);
        default: return launch_phase<kUpdate>(p, st);
    }
}

cudaError_t launch_tf32_split(const MatDev* mats, const MatTf32* tf32, int count, int max_tiles, cudaStream_t st) {
    if (count == 0 || max_tiles == 0) return cudaSuccess;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(max_tiles), unsigned(count));
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    return cudaLaunchKernelEx(&cfg, tf32_split_kernel, mats, tf32);
}

}  // namespace slorr
