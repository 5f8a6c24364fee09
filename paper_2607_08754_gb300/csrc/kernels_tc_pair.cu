// Grouped persistent tensor-core GEMM on CTA pairs (tcgen05 cta_group::2) for
// the three phases of a Polar Express step (Sec. 3 "Computing the polar
// factor"): Gram A = X X^T, Poly M = a I + b A + c A A, Update X' = M X, over
// every matrix of the weight set.  Two launch modes:
//   per-phase   one launch per phase and step (3 T launches); pair q runs
//               items q, q + npairs, ...; the launch boundary orders phases.
//   dataflow    one launch for every phase of every step.  Pair q runs its
//               own list of the host's plan, in order.  Each epilogue warp of
//               both CTAs adds 1 to its matrix's completion count once its
//               part of an item is stored (after a GPU-scope fence), and a TMA
//               producer waits (acquire, bounded) until the count reaches the
//               item's threshold -- every item of the matrix's earlier (step,
//               phase) groups -- before copying its operands.  So a matrix's
//               Poly tiles start as soon as its own Gram tiles are stored,
//               and the phases of different matrices overlap.  The plan lists
//               each pair's items in an order in which every item comes after
//               the items it waits for (see build_dataflow in api.cu), and all
//               pairs are resident, so the launch cannot deadlock.
//
// bf16 hi/lo operand mode (PairCfg<..., true>, per-phase launches): every
// product takes three products into the same accumulator -- the operands' hi
// parts, the A operand's lo part with B's hi part, A's hi part with B's lo
// part, one after the other for each K block (k_pass picks the tensor maps of
// each main-loop block) -- and the epilogues store hi and lo parts of A, M
// and X'.
//
// A cluster of two CTAs on two SMs computes one 256 x 256 tile.  CTA r of the
// pair holds rows [128 r, 128 r + 128) of the tile's A operand and columns
// [nsz/2 r, nsz/2 (r + 1)) of its B operand in shared memory, and rows
// [128 r, 128 r + 128) of the fp32 accumulator in its own tensor memory; one
// thread of the even CTA issues M = 256 UMMAs that read both CTAs' operands and
// write both CTAs' accumulators.  Each SM therefore moves the same bytes per
// FLOP as a single-CTA 256 x 256 tile, while a tile's accumulator takes only
// 256 TMEM columns per SM: two of them fit, so a tile's epilogue overlaps the
// next tile's main loop.
//
// Roles (192 threads per CTA; 320 for Poly and the dataflow launch):
//   warp 0 lane 0   TMA producer (both CTAs): waits for a stage to be free and
//                   loads its CTA's A rows and B half into its own shared
//                   memory, counting the bytes on the even CTA's stage barrier
//                   (the cta_group::2 form of the tensor copy);
//   warp 1          allocates the pair's TMEM (with the peer); lane 0 of the
//                   even CTA "arms" each stage barrier with the bytes of both
//                   CTAs' copies one ring ahead (as soon as the stage's current
//                   data has landed), issues the pair UMMAs, and multicasts
//                   each stage release and each tile completion to both CTAs;
//   warps 2..       epilogue (both CTAs): 128 rows of the tile from TMEM, one
//                   warp (two for Poly, each taking half of the columns) per
//                   32-row TMEM lane quadrant, each 32 x 32 chunk staged in
//                   the warp's shared-memory buffer so that global stores (and
//                   Poly's loads of A) move 8 rows x 64 bytes per instruction;
//                   then release the accumulator slot on the even CTA's barrier
//                   (and, in the dataflow launch, count the item as done).
// A stage is released only by a commit the MMA thread issues after arming the
// stage's next phase, so every copy of either CTA is counted on a phase the
// MMA thread armed; on a timeout that thread waits (bounded) for the last
// armed phase of every stage, and the exit cluster barrier keeps the odd CTA
// alive until then.  Every wait is bounded; a CTA that gives up sets the
// abort flag of both CTAs.  The only unbounded waits are the two cluster
// barriers at entry and exit, which every thread reaches after finitely many
// bounded waits.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <atomic>

#include "tc_common.cuh"

namespace slorr {
namespace {

using namespace tc;

template <int STAGES_, int EPIW_, bool SPLIT_ = false>
struct PairCfg {
    static constexpr int BK = kPairBK;                    // two 128-byte swizzle atoms of K
    static constexpr int STAGES = STAGES_;
    static constexpr bool kSplit = SPLIT_;                // bf16 hi/lo operands: three products per K block
    static constexpr int kSlots = 2;                      // accumulators per CTA in TMEM
    static constexpr int kABytes = kBM * BK * 2;          // this CTA's 128 rows of A
    static constexpr int kBBytes = 128 * BK * 2;          // this CTA's half of B (a 128-row box, <= 128 used)
    static constexpr uint32_t kAtomBytes = 128 * 128;     // one 128-row swizzle atom column (64 elements wide)
    static constexpr uint32_t kMnLbo = uint32_t(BK) * 128;  // MN-major: 64-element MN chunks this far apart
    static constexpr int kAccCols = kBNMax;               // fp32 TMEM columns of one accumulator
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kEpiWarps = EPIW_;               // 4, or 8: two per TMEM lane quadrant
    static_assert(EPIW_ == 4 || EPIW_ == 8, "epilogue warps");
    static constexpr int kThreads = 64 + 32 * kEpiWarps;
    static constexpr uint32_t kKLayout = 2u;              // SWIZZLE_128B
    static constexpr uint32_t kKSbo = 8 * 128;            // 8-row groups of 128-byte rows
    static constexpr uint32_t kTmemCols = uint32_t(kSlots) * uint32_t(kAccCols);
    static constexpr size_t kBarrierBytes = 512;
    static constexpr size_t kEpiBytes = size_t(kEpiWarps) * kStageWarpBytes;  // epilogue staging
    static constexpr size_t kSmemBytes = size_t(STAGES) * kStageBytes + 1024 /*align*/ + kBarrierBytes + kEpiBytes;
    static_assert((2 * STAGES + 2 * kSlots + 1) * 8 + 16 <= kBarrierBytes, "barrier area");
    static_assert(kSmemBytes <= 232448, "shared memory budget");
    static_assert(kTmemCols <= 512, "tensor memory budget");
};
// Ring depth (a build-time tuning knob): 3 stages of 64 KB.
#ifndef SLORR_PAIR_STAGES
#define SLORR_PAIR_STAGES 3
#endif
// Two accumulators per CTA (the tile epilogue overlaps the next main loop);
// the Poly epilogue, which also reads b A, takes 8 warps, the others 4 (more
// polling warps slow the producer and MMA threads of the long-K phases).
using PairCfg2 = PairCfg<SLORR_PAIR_STAGES, 4>;
using PairCfg2Wide = PairCfg<SLORR_PAIR_STAGES, 8>;
// bf16 hi/lo mode: the kernels that run three products per product and store
// low parts.  The mode runs per-phase launches only (a dataflow kernel with
// every phase's epilogue spills registers).
using PairCfg2Split = PairCfg<SLORR_PAIR_STAGES, 4, true>;
using PairCfg2WideSplit = PairCfg<SLORR_PAIR_STAGES, 8, true>;
static_assert(PairCfg2Wide::kEpiWarps == kDataflowEpiWarps, "the dataflow plan counts 2 x 8 warps per item");

struct PairSmem {
    uint8_t* stages;
    uint8_t* epi;      // kStageWarpBytes per epilogue warp
    uint64_t* full;    // even CTA: both CTAs' copies of the stage landed
    uint64_t* empty;   // stage consumed by the pair UMMAs (multicast commit)
    uint64_t* tfull;   // accumulator slot complete (multicast commit)
    uint64_t* tempty;  // even CTA: both CTAs' epilogues released the slot
    uint64_t* drain;
    uint32_t* tmem_slot;
    volatile int* abort;
    volatile int* never;  // stays 0: drain waits ignore the abort flag
    uint32_t peer;        // cluster rank of the other CTA
};

__device__ __forceinline__ void record_timeout(const GemmLaunch& p, const PairSmem& s) {
    *s.abort = 1;
    ptx::st_cluster_u32(ptx::mapa(ptx::smem_u32(const_cast<int*>(s.abort)), s.peer), 1u);
    atomicOr(p.status, kStatusTimeout);
}

// The items a CTA pair runs, in order: its range of the dataflow plan, or
// every npairs-th item of a per-phase launch.  A dataflow launch of fewer
// steps than the plan (slorr_run_steps) skips the later steps' items; every
// role skips the same ones.
template <int PH>
struct PairItems {
    int first, end, stride;
    __device__ PairItems(const GemmLaunch& p, int pair, int npairs) {
        if constexpr (PH == kAnyPhase) {
            first = p.pair_begin[pair];
            end = p.pair_begin[pair + 1];
            stride = 1;
        } else {
            first = pair;
            end = p.num_items;
            stride = npairs;
        }
    }
};

// The first index >= idx (in steps of `stride`, below `end`) whose item runs.
template <int PH>
__device__ __forceinline__ int next_running(const GemmLaunch& p, int idx, int end, int stride) {
    if constexpr (PH == kAnyPhase)
        while (idx < end && int(p.items[idx].step) >= p.steps) idx += stride;
    return idx;
}

// Dataflow launch: waits until the completion count of the item's matrix
// reaches the item's threshold.  The acquire load makes every store the
// counted epilogue warps made before their (fenced) increments visible to
// this thread.  Gives up on this CTA's abort flag, on a timeout recorded
// anywhere in the launch (the status word), or after the launch's budget.
// *seen receives the count that satisfied the wait.
__device__ __forceinline__ bool wait_done(const GemmLaunch& p, const PairSmem& s, const GemmItem& it,
                                          uint32_t* seen = nullptr) {
    if (it.wait == 0) return true;
    const uint32_t* c = p.done + it.mat;
    uint32_t v = ptx::ld_acquire_gpu(c);
    if (v >= it.wait) {
        if (seen) *seen = v;
        return true;
    }
    const uint64_t t0 = ptx::globaltimer();
    for (uint32_t i = 1;; ++i) {
        __nanosleep(32);
        v = ptx::ld_acquire_gpu(c);
        if (v >= it.wait) {
            if (seen) *seen = v;
            return true;
        }
        if ((i & 15u) == 0u) {
            if (*s.abort) return false;
            if (ptx::ld_relaxed_gpu(p.status) & kStatusTimeout) return false;
            if (ptx::globaltimer() - t0 > p.timeout_ns) return false;
        }
    }
}

// Diagonal tiles of the symmetric products (Gram A = X X^T, Poly A A): with
// tm == tn and a full 256 x 256 tile, each CTA's A rows and B columns are the
// same 128 rows of the same matrix, so they are copied once and both UMMA
// operands read them (the B descriptor points at the A half).  Not in bf16
// hi/lo mode, whose cross products take different parts for A and B.
template <class C, int PH>
__device__ __forceinline__ bool shared_operand(const GemmItem& it) {
    return !C::kSplit && item_phase<PH>(it) != kUpdate && it.tm == it.tn && it.msz == 2 * kBM &&
           it.nsz == kBNMax;
}

// Bytes one CTA of the pair copies per stage of a tile: its A rows, unless they
// lie beyond the matrix (the UMMA rows they would feed are never stored), and
// its half of the B columns, unless they are its A rows (shared_operand).
template <class C, int PH>
__device__ __forceinline__ uint32_t pair_stage_bytes(const GemmItem& it, int rank) {
    const uint32_t a = rank * kBM < it.msz ? uint32_t(C::kABytes) : 0u;
    return shared_operand<C, PH>(it) ? a : a + uint32_t(C::kBBytes);
}

template <class C, int PH>
__device__ void pair_producer(const GemmLaunch& p, const PairSmem& s, int rank, const PairItems<PH>& seq) {
    int stage = 0;
    uint32_t phase = 0;
    const uint32_t even_full = ptx::mapa(ptx::smem_u32(s.full), 0);
    // the last completion count this thread acquired, and of which matrix:
    // an item it already covers needs no new acquire
    int seen_mat = -1;
    uint32_t seen = 0;
    for (int idx = next_running<PH>(p, seq.first, seq.end, seq.stride); idx < seq.end;
         idx = next_running<PH>(p, idx + seq.stride, seq.end, seq.stride)) {
        const GemmItem it = p.items[idx];
        // Dataflow: the item's operands are complete once its matrix's earlier
        // phases are; the proxy fence orders those generic-proxy stores, now
        // visible to this thread, before its tensor copies read them.
        if constexpr (PH == kAnyPhase) {
            if (it.wait != 0 && !(int(it.mat) == seen_mat && seen >= it.wait)) {
                if (!wait_done(p, s, it, &seen)) {
                    record_timeout(p, s);
                    return;
                }
                ptx::fence_proxy_async_global();
                seen_mat = it.mat;
            }
        }
        const PhaseInfo pi = phase_info<C, PH>(p, it);
        const bool load_a = rank * kBM < it.msz;
        const bool load_b = !shared_operand<C, PH>(it);
        int kb_begin, kb_end;
        split_range(it, pi.nkb, &kb_begin, &kb_end);
        for (int kb = kb_begin; kb < kb_end; ++kb) {
            if (!ptx::mbar_wait(&s.empty[stage], phase ^ 1u, s.abort, p.timeout_ns)) {
                record_timeout(p, s);
                return;
            }
            uint8_t* sa = s.stages + size_t(stage) * C::kStageBytes;
            uint8_t* sb = sa + C::kABytes;
            const KPass kp = k_pass<C>(pi, kb);
            const int k = kp.kr * C::BK;
            const uint32_t bar = even_full + uint32_t(stage * 8);
            // one 3-D box per operand half: 128 rows (y) of two 64-element
            // chunks (z) of each row.  K-major: rows are MN, chunks are K;
            // MN-major: rows are K, chunks are MN.
            if (load_a) {
                const int mn = it.tm * (2 * kBM) + rank * kBM;
                if (!a_mn_at<PH>(pi, it, kp.kr))
                    ptx::tma_load_3d_pair(sa, kp.mapA, bar, 0, mn, k / 64);
                else
                    ptx::tma_load_3d_pair(sa, kp.mapA, bar, 0, k, mn / 64);
            }
            // B columns: this CTA's half, nsz / 2 = 64 or 128 (a 64-wide half
            // takes the same box; the UMMA reads its first 64)
            if (load_b) {
                const int mn = it.tn * kBNMax + rank * (it.nsz / 2);
                if (!b_mn_at<PH>(pi, it, kp.kr))
                    ptx::tma_load_3d_pair(sb, kp.mapB, bar, 0, mn, k / 64);
                else
                    ptx::tma_load_3d_pair(sb, kp.mapB, bar, 0, k, mn / 64);
            }
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
}

// Walks this pair's (tile, K block) sequence; the MMA thread keeps one cursor
// STAGES K blocks ahead of the one it consumes, to arm stage barriers.
template <class C, int PH>
struct KCursor {
    const GemmLaunch* p;
    int idx, end, stride, kb, nkb;
    uint32_t bytes;  // bytes both CTAs copy for the current K block
    __device__ void load() {
        idx = next_running<PH>(*p, idx, end, stride);
        if (idx < end) {
            const GemmItem it = p->items[idx];
            int b, e;
            split_range(it, phase_info<C, PH>(*p, it).nkb, &b, &e);
            nkb = e - b;
            bytes = pair_stage_bytes<C, PH>(it, 0) + pair_stage_bytes<C, PH>(it, 1);
        }
    }
    __device__ KCursor(const GemmLaunch& gp, const PairItems<PH>& seq)
        : p(&gp), idx(seq.first), end(seq.end), stride(seq.stride), kb(0), nkb(0), bytes(0) {
        load();
    }
    __device__ bool valid() const { return idx < end; }
    __device__ void next() {
        if (++kb == nkb) {
            kb = 0;
            idx += stride;
            load();
        }
    }
};

template <bool BF16, class C, int PH>
__device__ void pair_mma(const GemmLaunch& p, const PairSmem& s, uint32_t tmem_base, const PairItems<PH>& seq) {
    int armed_parity[C::STAGES];
#pragma unroll
    for (int i = 0; i < C::STAGES; ++i) armed_parity[i] = -1;
    // Arm the first ring: phase 0 of every stage the sequence reaches.
    KCursor<C, PH> arm(p, seq);
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
    for (int idx = next_running<PH>(p, seq.first, seq.end, seq.stride); idx < seq.end && ok;
         idx = next_running<PH>(p, idx + seq.stride, seq.end, seq.stride), ++local) {
        const GemmItem it = p.items[idx];
        const PhaseInfo pi = phase_info<C, PH>(p, it);
        const int slot = local % C::kSlots;
        const uint32_t tphase = uint32_t(local / C::kSlots) & 1u;
        if (!ptx::mbar_wait<true>(&s.tempty[slot], tphase ^ 1u, s.abort, p.timeout_ns)) {
            record_timeout(p, s);
            ok = false;
            break;
        }
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem_base + uint32_t(slot * C::kAccCols);
        int kb_begin, kb_end;
        split_range(it, pi.nkb, &kb_begin, &kb_end);
        for (int kb = kb_begin; kb < kb_end; ++kb) {
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
            ptx::tc_fence_after();
            const uint32_t a0 = ptx::smem_u32(s.stages + size_t(stage) * C::kStageBytes);
            const uint32_t b0 = shared_operand<C, PH>(it) ? a0 : a0 + C::kABytes;
            const int kr = k_pass<C>(pi, kb).kr;
            const bool a_mn = a_mn_at<PH>(pi, it, kr);
            const bool b_mn = b_mn_at<PH>(pi, it, kr);
            const uint32_t id = ptx::idesc_f16(2 * kBM, it.nsz, BF16, a_mn, b_mn);
#pragma unroll
            for (int kk = 0; kk < C::BK / 16; ++kk) {
                const uint32_t acc = (kb != kb_begin || kk != 0) ? 1u : 0u;
                ptx::umma_f16_pair(d_tmem, operand_desc<C>(a0, kk, a_mn), operand_desc<C>(b0, kk, b_mn), id, acc);
            }
            issued_any = true;
            ptx::umma_commit_pair_mc(&s.empty[stage], 0x3);
            if (++stage == C::STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        ptx::umma_commit_pair_mc(&s.tfull[slot], 0x3);
    }
    if (!ok) {
        if (issued_any) {
            // No UMMA may still be writing either CTA's TMEM when it is released.
            ptx::umma_commit_pair_mc(s.drain, 0x1);
            ptx::mbar_wait(s.drain, 0u, s.never, p.timeout_ns);
        }
        // Every copy either CTA issued was counted on an armed phase: wait
        // (bounded) for the last armed phase of each stage before exit.
        for (int i = 0; i < C::STAGES; ++i)
            if (armed_parity[i] >= 0) ptx::mbar_wait(&s.full[i], uint32_t(armed_parity[i]), s.never, p.timeout_ns);
    }
}

template <bool BF16, class C, int PH>
__device__ void pair_epilogue(const GemmLaunch& p, const PairSmem& s, uint32_t tmem_base, int rank,
                              const PairItems<PH>& seq, int warp, int lane) {
    const int quad = warp & 3;             // TMEM lanes [32 quad, 32 quad + 32) (hardware rule)
    const int ngroups = C::kEpiWarps / 4;  // warps per lane quadrant, splitting the columns
    const int group = (warp - 2) / 4;
    uint8_t* sbuf = s.epi + (warp - 2) * kStageWarpBytes;
    int local = 0;
    const uint32_t even_tempty = ptx::mapa(ptx::smem_u32(s.tempty), 0);
    for (int idx = next_running<PH>(p, seq.first, seq.end, seq.stride); idx < seq.end;
         idx = next_running<PH>(p, idx + seq.stride, seq.end, seq.stride), ++local) {
        const GemmItem it = p.items[idx];
        const MatDev& md = p.mats[it.mat];
        const int slot = local % C::kSlots;
        const uint32_t tphase = uint32_t(local / C::kSlots) & 1u;
        int ok = 1;
        if (lane == 0) {
            ok = ptx::mbar_wait(&s.tfull[slot], tphase, s.abort, p.timeout_ns) ? 1 : 0;
            // Poly reads b A with plain loads: acquire A's completion count in
            // this thread too (the producer already saw it reached).
            if constexpr (PH == kAnyPhase)
                if (ok && it.phase == kPoly && !wait_done(p, s, it)) ok = 0;
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) record_timeout(p, s);
            break;
        }
        ptx::tc_fence_after();
        if (rank * kBM < it.msz) {
            const int row0 = it.tm * (2 * kBM) + rank * kBM;
            const uint32_t t_row = tmem_base + (uint32_t(quad * 32) << 16) + uint32_t(slot * C::kAccCols);
            const int per = it.nsz / 32 / ngroups;  // 32-column chunks per warp
            const int parts = it.ksplit >> 8;
            if (parts <= 1) {
                store_rows<BF16, PH, true, C::kSplit>(p, it, md, row0, t_row, quad, lane, group * per,
                                                      (group + 1) * per, nullptr, 1, 0, sbuf);
            } else if (PH != kPoly && PH != kUpdate &&
                       split_partial_is_last(p, it, rank, quad, group, lane, t_row, group * per, (group + 1) * per)) {
                // split K (Gram): direct stores, since the last part's sum is a
                // serial step, which the staging round trip lengthens (small
                // sets, ResNet-18 Gram +7%)
                store_rows<BF16, PH, false, C::kSplit>(p, it, md, row0, t_row, quad, lane, group * per,
                                                       (group + 1) * per, p.split_part + size_t(it.sid) * 65536,
                                                       parts, rank * kBM + quad * 32 + lane);
            }
        }
        // The slot may be overwritten once this warp's TMEM loads are done
        // (tcgen05.wait::ld above); the stores need no ordering with the
        // next UMMAs, so the arrive is relaxed.
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) {
            ptx::mbar_arrive_cluster_relaxed(even_tempty + uint32_t(slot * 8));
            // Dataflow: publish this warp's part of the item (every lane's
            // stores happen before the fence through the warp barrier above).
            if constexpr (PH == kAnyPhase) {
                __threadfence();
                atomicAdd(p.done + it.mat, 1u);
            }
        }
    }
}

template <bool BF16, class C, int PH>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(C::kThreads, 1)
    tc_pair_kernel(const __grid_constant__ GemmLaunch p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    PairSmem s;
    s.stages = base;
    s.epi = base + size_t(C::STAGES) * C::kStageBytes + C::kBarrierBytes;
    s.full = reinterpret_cast<uint64_t*>(base + size_t(C::STAGES) * C::kStageBytes);
    s.empty = s.full + C::STAGES;
    s.tfull = s.empty + C::STAGES;
    s.tempty = s.tfull + C::kSlots;
    s.drain = s.tempty + C::kSlots;
    s.tmem_slot = reinterpret_cast<uint32_t*>(s.drain + 1);
    s.abort = reinterpret_cast<volatile int*>(s.tmem_slot + 1);
    s.never = s.abort + 1;
    const int rank = int(ptx::cluster_ctarank());
    s.peer = uint32_t(rank ^ 1);
    const int pair = blockIdx.x / 2, npairs = gridDim.x / 2;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const PairItems<PH> seq(p, pair, npairs);

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::STAGES; ++i) {
            ptx::mbar_init(&s.full[i], 1);
            ptx::mbar_init(&s.empty[i], 1);
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
    if (warp == 0 && lane == 0 && seq.first < seq.end) {
        const PhaseInfo pi = phase_info<C, PH>(p, p.items[seq.first]);
        ptx::prefetch_tmap(pi.mapA);
        ptx::prefetch_tmap(pi.mapB);
    }
    if (warp == 1) {
        ptx::tmem_alloc_pair(s.tmem_slot, C::kTmemCols);
        ptx::tmem_relinquish_pair();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // barriers initialised and TMEM allocated in both CTAs
    ptx::tc_fence_after();
    const uint32_t tmem_base = *s.tmem_slot;
    // The UMMAs address both CTAs' accumulators with the even CTA's TMEM
    // address: the two allocations must agree, else no work is done.
    const uint32_t peer_base = ptx::ld_cluster_u32(ptx::mapa(ptx::smem_u32(s.tmem_slot), s.peer));
    // Under programmatic dependent launch everything above overlapped the
    // previous kernel's tail; wait for its results before any role starts.
    ptx::griddep_wait();
    ptx::griddep_launch_dependents();
    if (peer_base != tmem_base) {
        if (threadIdx.x == 0) atomicOr(p.status, kStatusInternal);
    } else if (warp == 0) {
        if (lane == 0) pair_producer<C, PH>(p, s, rank, seq);
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) pair_mma<BF16, C, PH>(p, s, tmem_base, seq);
        __syncwarp();
    } else {
        pair_epilogue<BF16, C, PH>(p, s, tmem_base, rank, seq, warp, lane);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // no remote arrive, UMMA or copy of either CTA is outstanding
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc_pair(tmem_base, C::kTmemCols);
    }
}

// Co-resident CTA pairs of one kernel configuration on each device, found
// once per device (the function attribute is per device, too).  Concurrent
// first queries on one device may both run; they store the same value.
constexpr int kMaxDevices = 64;

template <bool BF16, class C, int PH>
cudaError_t max_pairs_of(int num_sms, int* out) {
    static std::atomic<int> cache[kMaxDevices];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    int max_pairs = cache[dev].load(std::memory_order_acquire);
    if (max_pairs == 0) {
        e = cudaFuncSetAttribute(tc_pair_kernel<BF16, C, PH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(C::kSmemBytes));
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t probe = {};
        probe.gridDim = dim3(unsigned(2 * (num_sms / 2)));
        probe.blockDim = dim3(C::kThreads);
        probe.dynamicSmemBytes = C::kSmemBytes;
        int clusters = 0;
        e = cudaOccupancyMaxActiveClusters(&clusters, tc_pair_kernel<BF16, C, PH>, &probe);
        if (e != cudaSuccess) return e;
        if (clusters < 1) return cudaErrorInvalidConfiguration;
        max_pairs = clusters < num_sms / 2 ? clusters : num_sms / 2;
        cache[dev].store(max_pairs, std::memory_order_release);
    }
    *out = max_pairs;
    return cudaSuccess;
}

// Per-phase launches: min(items, co-resident pairs) pairs.  Dataflow launch:
// exactly the plan's `npairs` pairs, which must all be resident at once (a
// pair may wait for items of any other), so a plan for more pairs than fit is
// refused.
template <bool BF16, class C, int PH>
cudaError_t launch_pair_cfg(const GemmLaunch& p, int num_sms, cudaStream_t st, int npairs) {
    int max_pairs = 0;
    cudaError_t e = max_pairs_of<BF16, C, PH>(num_sms, &max_pairs);
    if (e != cudaSuccess) return e;
    if constexpr (PH == kAnyPhase) {
        if (npairs < 1 || npairs > max_pairs) return cudaErrorInvalidConfiguration;
    } else {
        npairs = p.num_items < max_pairs ? p.num_items : max_pairs;
    }
    return launch_kernel(tc_pair_kernel<BF16, C, PH>, unsigned(2 * npairs), C::kThreads, C::kSmemBytes, st,
                         p.pdl != 0, p);
}

template <bool BF16>
cudaError_t launch_pair_bf(const GemmLaunch& p, int num_sms, cudaStream_t st, int phase, int npairs) {
    switch (phase) {
        case kGram: return launch_pair_cfg<BF16, PairCfg2, kGram>(p, num_sms, st, npairs);
        case kPoly: return launch_pair_cfg<BF16, PairCfg2Wide, kPoly>(p, num_sms, st, npairs);
        case kUpdate: return launch_pair_cfg<BF16, PairCfg2, kUpdate>(p, num_sms, st, npairs);
        default: return launch_pair_cfg<BF16, PairCfg2Wide, kAnyPhase>(p, num_sms, st, npairs);
    }
}

cudaError_t launch_pair_split(const GemmLaunch& p, int num_sms, cudaStream_t st, int phase, int npairs) {
    switch (phase) {
        case kGram: return launch_pair_cfg<true, PairCfg2Split, kGram>(p, num_sms, st, npairs);
        case kPoly: return launch_pair_cfg<true, PairCfg2WideSplit, kPoly>(p, num_sms, st, npairs);
        case kUpdate: return launch_pair_cfg<true, PairCfg2Split, kUpdate>(p, num_sms, st, npairs);
        default: return cudaErrorInvalidValue;  // no dataflow launch in this mode
    }
}

}  // namespace

cudaError_t launch_gemm_tc_pair(const GemmLaunch& p, int elem, int num_sms, cudaStream_t st, int phase,
                                int npairs) {
    if (p.num_items == 0) return cudaSuccess;
    if (p.split) {
        if (elem != kBF16) return cudaErrorInvalidValue;  // hi/lo parts are bf16
        return launch_pair_split(p, num_sms, st, phase, npairs);
    }
    return elem == kBF16 ? launch_pair_bf<true>(p, num_sms, st, phase, npairs)
                         : launch_pair_bf<false>(p, num_sms, st, phase, npairs);
}

cudaError_t tc_pair_dataflow_capacity(int elem, int num_sms, int* pairs) {
    *pairs = 0;
    return elem == kBF16 ? max_pairs_of<true, PairCfg2Wide, kAnyPhase>(num_sms, pairs)
                         : max_pairs_of<false, PairCfg2Wide, kAnyPhase>(num_sms, pairs);
}

}  // namespace slorr
