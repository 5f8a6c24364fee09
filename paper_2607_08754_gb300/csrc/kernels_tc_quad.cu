// Grouped persistent tensor-core GEMM on clusters of two CTA pairs, for the
// same three phases of a Polar Express step as kernels_tc_pair.cu (Sec. 3
// "Computing the polar factor"): Gram A = X X^T, Poly M = a I + b A + c A A,
// Update X' = M X, over every matrix of the weight set in one launch.
//
// The pair kernel is bound by the rate at which TMA moves operands from L2
// into shared memory: a 256 x 256 tile reads 2 x 256 rows per K block.  Here a
// cluster of four CTAs -- pair 0 (ranks 0, 1) and pair 1 (ranks 2, 3) --
// computes a super-tile of two 256 x 256 tiles that share an operand: the same
// A rows (tiles (tm, tn0) and (tm, tn1)) or the same B columns (tiles
// (tm0, tn) and (tm1, tn)).  The shared operand is loaded once: CTA r and its
// counterpart r ^ 2 in the other pair each load half of it with a TMA
// multicast to both, so each SM reads 3/4 of the bytes per FLOP of a pair.
// Each pair then runs exactly as in the pair kernel: M = 256 UMMAs from its
// even CTA over both CTAs' operands, two accumulators per SM, an epilogue that
// overlaps the next tile.  A super-tile whose second tile is empty (an odd
// leftover) runs on pair 0 while pair 1 steps through the same K blocks idly.
//
// Synchronisation:
//   full[s]   (pair leaders) the bytes of the pair's copies of stage s; armed
//             by the leader's MMA thread one ring ahead (0 bytes when idle);
//             every copy of the cluster completes on the barrier of its
//             destination's pair leader (cta_group::2 copies, multicast ones
//             included);
//   empty[s]  (every CTA) two arrivals per phase: the stage-release commits
//             of both pairs' MMA threads, multicast to all four CTAs, so a
//             producer reloads a stage -- its own or, by multicast, its
//             counterpart's -- only once both pairs are done with it (an idle
//             pair releases phase k of a stage only after phase k - 1 was
//             released by both, which keeps the arrivals of each phase
//             paired);
//   tfull / tempty / drain: per pair, as in the pair kernel.
// Every copy therefore lands on a phase its destination's pair leader armed
// before the stage was released; on a timeout each leader drains its last
// armed phases, and the exit cluster barrier keeps all four CTAs alive until
// both have.  Every wait is bounded; a CTA that gives up sets the abort flag
// of all four CTAs.  The only unbounded waits are the two cluster barriers at
// entry and exit, which every thread reaches after finitely many bounded
// waits.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "tc_common.cuh"

namespace slorr {
namespace {

using namespace tc;

template <int STAGES_, int EPIW_>
struct QuadCfg {
    static constexpr int BK = 64;
    static constexpr int STAGES = STAGES_;
    static constexpr int kSlots = 2;                      // accumulators per CTA in TMEM
    static constexpr int kBoxBytes = 64 * BK * 2;         // one 64 x 64 box
    static constexpr int kABytes = kBM * BK * 2;          // this CTA's 128 rows of A
    static constexpr int kBBytes = (kBNMax / 2) * BK * 2; // this CTA's half of B (<= 128 rows)
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kEpiWarps = EPIW_;
    static constexpr int kThreads = 64 + 32 * kEpiWarps;
    static constexpr uint32_t kKLayout = 2u;              // SWIZZLE_128B
    static constexpr uint32_t kKSbo = 8 * BK * 2;
    static constexpr uint32_t kTmemCols = uint32_t(kSlots) * kAccCols;
    static constexpr size_t kBarrierBytes = 512;
    static constexpr size_t kSmemBytes = size_t(STAGES) * kStageBytes + 1024 /*align*/ + kBarrierBytes;
    static_assert(EPIW_ == 4 || EPIW_ == 8, "epilogue warps");
    static_assert((2 * STAGES + 2 * kSlots + 1) * 8 + 16 <= kBarrierBytes, "barrier area");
    static_assert(kSmemBytes <= 232448, "shared memory budget");
};
using QuadCfg4 = QuadCfg<6, 4>;   // Gram, Update
using QuadCfg8 = QuadCfg<6, 8>;   // Poly (its epilogue also reads b A)

struct QuadSmem {
    uint8_t* stages;
    uint64_t* full;    // pair leader: both CTAs' bytes of the stage landed
    uint64_t* empty;   // stage released by both pairs (two multicast commits)
    uint64_t* tfull;   // accumulator slot complete (commit multicast to the pair)
    uint64_t* tempty;  // pair leader: both CTAs' epilogues released the slot
    uint64_t* drain;
    uint32_t* tmem_slot;
    volatile int* abort;
    volatile int* never;  // stays 0: drain waits ignore the abort flag
    uint32_t rank;        // cluster rank: pair rank >> 1, role in the pair rank & 1
};

__device__ __forceinline__ void record_timeout(const GemmLaunch& p, const QuadSmem& s) {
    *s.abort = 1;
    const uint32_t a = ptx::smem_u32(const_cast<int*>(s.abort));
    for (uint32_t r = 0; r < 4; ++r)
        if (r != s.rank) ptx::st_cluster_u32(ptx::mapa(a, r), 1u);
    atomicOr(p.status, kStatusTimeout);
}

// Bytes one CTA of a pair receives per K block of tile `it` (its A rows unless
// they lie beyond the matrix, and its half of the B columns).
template <class C>
__device__ __forceinline__ uint32_t cta_stage_bytes(const GemmItem& it, int prank) {
    return (prank * kBM < it.msz ? uint32_t(C::kABytes) : 0u) + uint32_t(it.nsz / 2) * C::BK * 2;
}

// One super-tile as seen by pair `pair_id`.
struct Super {
    GemmItem mine;   // this pair's tile (msz = 0: none)
    bool present;    // this pair has a tile
    bool share_a;    // both tiles have the same A rows
    bool share_b;    // both tiles have the same B columns
};

__device__ __forceinline__ Super super_info(const GemmLaunch& p, int idx, int pair_id) {
    const GemmItem a = p.items[2 * idx], b = p.items[2 * idx + 1];
    Super su;
    su.mine = pair_id ? b : a;
    su.present = su.mine.msz != 0;
    const bool both = b.msz != 0;
    su.share_a = both && a.tm == b.tm;
    su.share_b = both && !su.share_a && a.tn == b.tn;
    return su;
}

template <class C>
__device__ void quad_producer(const GemmLaunch& p, const QuadSmem& s, int cl, int ncl) {
    const int rank = int(s.rank), pair_id = rank >> 1, prank = rank & 1;
    const uint32_t leader_full = ptx::mapa(ptx::smem_u32(s.full), uint32_t(rank & ~1));
    const uint16_t mc = uint16_t((1u << rank) | (1u << (rank ^ 2)));  // this CTA and its counterpart
    int stage = 0;
    uint32_t phase = 0;
    for (int idx = cl; idx < p.num_items; idx += ncl) {
        const Super su = super_info(p, idx, pair_id);
        const GemmItem it = su.mine;
        const PhaseInfo pi = phase_info<C>(p, p.items[2 * idx]);
        const bool load_a = su.present && prank * kBM < it.msz;
        const int bhalf = it.nsz / 2;  // 64 or 128 rows of B per CTA
        for (int kb = 0; kb < pi.nkb; ++kb) {
            if (!ptx::mbar_wait(&s.empty[stage], phase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                return;
            }
            if (su.present) {
                uint8_t* sa = s.stages + size_t(stage) * C::kStageBytes;
                uint8_t* sb = sa + C::kABytes;
                const int k = kb * C::BK;
                const uint32_t bar = leader_full + uint32_t(stage * 8);
                // box coordinates are (inner, outer): (k, mn) for K-major, (mn, k) for MN-major
                if (load_a)
                    for (int b = 0; b < 2; ++b) {
                        if (su.share_a && b != pair_id) continue;  // the counterpart loads it
                        const int mn = it.tm * (2 * kBM) + prank * kBM + b * 64;
                        const int x = pi.a_mn ? mn : k, y = pi.a_mn ? k : mn;
                        if (su.share_a)
                            ptx::tma_load_2d_pair_mc(sa + b * C::kBoxBytes, pi.mapA, bar, x, y, mc);
                        else
                            ptx::tma_load_2d_pair(sa + b * C::kBoxBytes, pi.mapA, bar, x, y);
                    }
                for (int j = 0; j < bhalf / 64; ++j) {
                    if (su.share_b && (j & 1) != pair_id) continue;
                    const int mn = it.tn * kBNMax + prank * bhalf + j * 64;
                    const int x = pi.b_mn ? mn : k, y = pi.b_mn ? k : mn;
                    if (su.share_b)
                        ptx::tma_load_2d_pair_mc(sb + j * C::kBoxBytes, pi.mapB, bar, x, y, mc);
                    else
                        ptx::tma_load_2d_pair(sb + j * C::kBoxBytes, pi.mapB, bar, x, y);
                }
            }
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
}

// Walks this cluster's (super-tile, K block) sequence for one pair; the MMA
// thread keeps one cursor STAGES K blocks ahead to arm its stage barriers.
template <class C>
struct QCursor {
    const GemmLaunch* p;
    int idx, kb, nkb, step, pair_id;
    uint32_t bytes;  // bytes the pair's two CTAs receive for the current K block
    __device__ void load() {
        if (idx < p->num_items) {
            nkb = phase_info<C>(*p, p->items[2 * idx]).nkb;
            const Super su = super_info(*p, idx, pair_id);
            bytes = su.present ? cta_stage_bytes<C>(su.mine, 0) + cta_stage_bytes<C>(su.mine, 1) : 0u;
        }
    }
    __device__ QCursor(const GemmLaunch& gp, int first, int stride, int pid)
        : p(&gp), idx(first), kb(0), nkb(0), step(stride), pair_id(pid), bytes(0) {
        load();
    }
    __device__ bool valid() const { return idx < p->num_items; }
    __device__ void next() {
        if (++kb == nkb) {
            kb = 0;
            idx += step;
            load();
        }
    }
};

template <bool BF16, class C>
__device__ void quad_mma(const GemmLaunch& p, const QuadSmem& s, uint32_t tmem_base, int cl, int ncl) {
    const int pair_id = int(s.rank) >> 1;
    const uint16_t pair_mask = uint16_t(0x3u << (2 * pair_id));
    int armed_parity[C::STAGES];
#pragma unroll
    for (int i = 0; i < C::STAGES; ++i) armed_parity[i] = -1;
    QCursor<C> arm(p, cl, ncl, pair_id);
    for (int i = 0; i < C::STAGES && arm.valid(); ++i, arm.next()) {
        ptx::mbar_arrive_expect_tx(&s.full[i], arm.bytes);
        armed_parity[i] = 0;
    }
    int stage = 0;
    uint32_t phase = 0;
    int local = 0;
    bool ok = true;
    bool issued_any = false;
    if (p.test_stall) {
        // Failure-detection test: wait on the drain barrier, which nothing
        // arrives on before the end, so the bounded wait runs out.
        if (!ptx::mbar_wait(s.drain, 0u, s.abort, p.timeout_ns)) {
            record_timeout(p, s);
            ok = false;
        }
    }
    for (int idx = cl; idx < p.num_items && ok; idx += ncl) {
        const Super su = super_info(p, idx, pair_id);
        const GemmItem it = su.mine;
        const PhaseInfo pi = phase_info<C>(p, p.items[2 * idx]);
        const int slot = local % C::kSlots;
        const uint32_t tphase = uint32_t(local / C::kSlots) & 1u;
        if (su.present) {
            if (!ptx::mbar_wait<true>(&s.tempty[slot], tphase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            ptx::tc_fence_after();
        }
        const uint32_t idesc = ptx::idesc_f16(2 * kBM, it.nsz, BF16, pi.a_mn, pi.b_mn);
        const uint32_t d_tmem = tmem_base + uint32_t(slot * kAccCols);
        for (int kb = 0; kb < pi.nkb; ++kb) {
            if (!ptx::mbar_wait(&s.full[stage], phase, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                ok = false;
                break;
            }
            // This stage's data has landed, so its barrier is in its next phase:
            // arm it now for the K block one ring ahead.
            if (arm.valid()) {
                ptx::mbar_arrive_expect_tx(&s.full[stage], arm.bytes);
                armed_parity[stage] = int(phase ^ 1u);
                arm.next();
            }
            if (!su.present) {
                // Idle pair: its stage barriers complete at once (0 bytes), so
                // nothing else keeps its releases in step with the working
                // pair's.  Each phase of `empty` must collect one release from
                // each pair, so wait until the stage's previous phase has been
                // released by both before releasing this one.  (A working pair
                // always satisfies this already: its copies for this phase were
                // issued only after that release.)
                if (!ptx::mbar_wait(&s.empty[stage], phase ^ 1u, s.abort, p.timeout_ns)) {
                    record_timeout(p, s);
                    ok = false;
                    break;
                }
            }
            if (su.present) {
                ptx::tc_fence_after();
                const uint32_t a0 = ptx::smem_u32(s.stages + size_t(stage) * C::kStageBytes);
                const uint32_t b0 = a0 + C::kABytes;
#pragma unroll
                for (int kk = 0; kk < C::BK / 16; ++kk)
                    ptx::umma_f16_pair(d_tmem, operand_desc<C>(a0, kk, pi.a_mn), operand_desc<C>(b0, kk, pi.b_mn),
                                       idesc, (kb | kk) != 0 ? 1u : 0u);
                issued_any = true;
            }
            // released to all four CTAs: the other pair may load into this
            // pair's shared memory by multicast
            ptx::umma_commit_pair_mc(&s.empty[stage], 0xF);
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        if (su.present) {
            ptx::umma_commit_pair_mc(&s.tfull[slot], pair_mask);
            ++local;
        }
    }
    if (!ok) {
        if (issued_any) {
            // No UMMA may still be writing either CTA's TMEM when it is released.
            ptx::umma_commit_pair_mc(s.drain, uint16_t(1u << s.rank));
            ptx::mbar_wait(s.drain, 0u, s.never, p.timeout_ns);
        }
        // Every copy into this pair's CTAs was counted on an armed phase: wait
        // (bounded) for the last armed phase of each stage before exit.
        for (int i = 0; i < C::STAGES; ++i)
            if (armed_parity[i] >= 0) ptx::mbar_wait(&s.full[i], uint32_t(armed_parity[i]), s.never, p.timeout_ns);
    }
}

template <bool BF16, class C>
__device__ void quad_epilogue(const GemmLaunch& p, const QuadSmem& s, uint32_t tmem_base, int cl, int ncl,
                              int warp, int lane) {
    const int rank = int(s.rank), pair_id = rank >> 1, prank = rank & 1;
    const int quad = warp & 3;             // TMEM lanes [32 quad, 32 quad + 32) (hardware rule)
    const int ngroups = C::kEpiWarps / 4;  // warps per lane quadrant, splitting the columns
    const int group = (warp - 2) / 4;
    const uint32_t leader_tempty = ptx::mapa(ptx::smem_u32(s.tempty), uint32_t(rank & ~1));
    int local = 0;
    for (int idx = cl; idx < p.num_items; idx += ncl) {
        const Super su = super_info(p, idx, pair_id);
        if (!su.present) continue;
        const GemmItem it = su.mine;
        const MatDev& md = p.mats[it.mat];
        const int slot = local % C::kSlots;
        const uint32_t tphase = uint32_t(local / C::kSlots) & 1u;
        ++local;
        int ok = 1;
        if (lane == 0) ok = ptx::mbar_wait(&s.tfull[slot], tphase, s.abort, p.timeout_ns) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) record_timeout(p, s);
            break;
        }
        ptx::tc_fence_after();
        if (prank * kBM < it.msz) {
            const int row0 = it.tm * (2 * kBM) + prank * kBM;
            const uint32_t t_row = tmem_base + (uint32_t(quad * 32) << 16) + uint32_t(slot * kAccCols);
            const int per = it.nsz / 32 / ngroups;  // 32-column chunks per warp
            store_rows<BF16, 2>(p, it, md, row0, t_row, quad, lane, group * per, (group + 1) * per);
        }
        // The slot may be overwritten once this warp's TMEM loads are done.
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive_cluster_relaxed(leader_tempty + uint32_t(slot * 8));
    }
}

template <bool BF16, class C>
__global__ void __cluster_dims__(4, 1, 1) __launch_bounds__(C::kThreads, 1)
    tc_quad_kernel(const __grid_constant__ GemmLaunch p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    QuadSmem s;
    s.stages = base;
    s.full = reinterpret_cast<uint64_t*>(base + size_t(C::STAGES) * C::kStageBytes);
    s.empty = s.full + C::STAGES;
    s.tfull = s.empty + C::STAGES;
    s.tempty = s.tfull + C::kSlots;
    s.drain = s.tempty + C::kSlots;
    s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
    s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
    s.never = s.abort + 1;
    s.rank = ptx::cluster_ctarank();
    const int cl = blockIdx.x / 4, ncl = gridDim.x / 4;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::STAGES; ++i) {
            ptx::mbar_init(&s.full[i], 1);
            ptx::mbar_init(&s.empty[i], 2);
        }
        for (int i = 0; i < C::kSlots; ++i) {
            ptx::mbar_init(&s.tfull[i], 1);
            ptx::mbar_init(&s.tempty[i], 2 * C::kEpiWarps);
        }
        ptx::mbar_init(s.drain, 1);
        *s.abort = 0;
        *s.never = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 0 && lane == 0 && cl < p.num_items) {
        const PhaseInfo pi = phase_info<C>(p, p.items[2 * cl]);
        ptx::prefetch_tmap(pi.mapA);
        ptx::prefetch_tmap(pi.mapB);
    }
    if (warp == 1) {
        ptx::tmem_alloc_pair(s.tmem_slot, C::kTmemCols);
        ptx::tmem_relinquish_pair();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // barriers initialised and TMEM allocated in all four CTAs
    ptx::tc_fence_after();
    const uint32_t tmem_base = *s.tmem_slot;
    // Each pair's UMMAs address both of its CTAs' accumulators with the even
    // CTA's TMEM address: the pair's allocations must agree, else no work is
    // done (every CTA reads all four, so all take the same decision).
    bool agree = true;
    for (uint32_t r = 0; r < 4; r += 2)
        agree = agree && ptx::ld_cluster_u32(ptx::mapa(ptx::smem_u32(s.tmem_slot), r)) ==
                             ptx::ld_cluster_u32(ptx::mapa(ptx::smem_u32(s.tmem_slot), r + 1));
    if (!agree) {
        if (threadIdx.x == 0) atomicOr(p.status, kStatusInternal);
    } else if (warp == 0) {
        if (lane == 0) quad_producer<C>(p, s, cl, ncl);
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0 && (s.rank & 1u) == 0) quad_mma<BF16, C>(p, s, tmem_base, cl, ncl);
        __syncwarp();
    } else {
        quad_epilogue<BF16, C>(p, s, tmem_base, cl, ncl, warp, lane);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // no remote arrive, UMMA or copy of any CTA is outstanding
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc_pair(tmem_base, C::kTmemCols);
    }
}

template <bool BF16, class C>
cudaError_t launch_quad_cfg(const GemmLaunch& p, int num_sms, cudaStream_t st) {
    static int max_clusters = 0;
    if (max_clusters == 0) {
        cudaError_t e = cudaFuncSetAttribute(tc_quad_kernel<BF16, C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             int(C::kSmemBytes));
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t probe = {};
        probe.gridDim = dim3(unsigned(4 * (num_sms / 4)));
        probe.blockDim = dim3(C::kThreads);
        probe.dynamicSmemBytes = C::kSmemBytes;
        int clusters = 0;
        e = cudaOccupancyMaxActiveClusters(&clusters, tc_quad_kernel<BF16, C>, &probe);
        if (e != cudaSuccess) return e;
        if (clusters < 1) return cudaErrorInvalidConfiguration;
        max_clusters = clusters < num_sms / 4 ? clusters : num_sms / 4;
    }
    const int ncl = p.num_items < max_clusters ? p.num_items : max_clusters;
    tc_quad_kernel<BF16, C><<<4 * ncl, C::kThreads, C::kSmemBytes, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_tc_quad(const GemmLaunch& p, int elem, int num_sms, cudaStream_t st) {
    if (p.num_items == 0) return cudaSuccess;
    const bool bf = elem == kBF16;
    if (p.phase == kPoly)
        return bf ? launch_quad_cfg<true, QuadCfg8>(p, num_sms, st) : launch_quad_cfg<false, QuadCfg8>(p, num_sms, st);
    return bf ? launch_quad_cfg<true, QuadCfg4>(p, num_sms, st) : launch_quad_cfg<false, QuadCfg4>(p, num_sms, st);
}

}  // namespace slorr
