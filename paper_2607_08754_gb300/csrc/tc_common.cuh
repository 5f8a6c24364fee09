// Pieces of the tensor-core GEMM kernel (kernels_tc_pair.cu: a CTA pair per
// 256 x 256 tile): 16-bit packing, the operand maps and orientation of each
// phase, the symmetric-tile rule, shared-memory operand descriptors and the
// epilogue of one 128-row block.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "internal.h"
#include "ptx.cuh"

namespace slorr {
namespace tc {

constexpr int kBM = 128;       // rows of one UMMA M tile (per CTA)
constexpr int kBNMax = 256;    // columns of a tile
constexpr int kAccCols = 256;  // fp32 TMEM columns of one 128 x 256 accumulator

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

// The kernel template's phase: kGram, kPoly or kUpdate for a per-phase launch
// (its epilogue and operand code compile for that phase alone), kAnyPhase for
// the dataflow launch (each item's own phase).
constexpr int kAnyPhase = -1;

template <int PH>
__device__ __forceinline__ int item_phase(const GemmItem& it) {
    if constexpr (PH >= 0)
        return PH;
    else
        return int(it.phase);
}

// The Polar Express step an item belongs to: its own (dataflow launch) or the
// launch's (per-phase launches).
template <int PH>
__device__ __forceinline__ int item_step(const GemmLaunch& p, const GemmItem& it) {
    if constexpr (PH >= 0)
        return p.step;
    else
        return int(it.step);
}

struct PhaseInfo {
    const void* mapA;
    const void* mapB;
    const void* mapAlo;  // bf16 hi/lo mode: the low parts of the A operand (else mapA)
    const void* mapBlo;  // and of the B operand (else mapB)
    int nkb;     // K blocks the tile's main loop runs (3 nkr in bf16 hi/lo mode)
    int nkr;     // K blocks of the product's K
    bool a_mn;   // A operand MN-major (else K-major)
    bool b_mn;   // B operand MN-major (else K-major)
};

// Tensor maps per matrix (kMapsPerMatrix of them, 128 bytes each): X0, X1,
// A, M, X0_lo, X1_lo, M_lo, A_lo.
__device__ __forceinline__ const void* xmap(const uint8_t* maps, int buf) { return maps + buf * 128; }
__device__ __forceinline__ const void* xlo_map(const uint8_t* maps, int buf) { return maps + (4 + buf) * 128; }

template <class C, int PH>
__device__ __forceinline__ PhaseInfo phase_info(const GemmLaunch& p, const GemmItem& it) {
    const MatDev& md = p.mats[it.mat];
    const uint8_t* maps = reinterpret_cast<const uint8_t*>(p.maps) + size_t(it.mat) * kMapsPerMatrix * 128;
    const bool tr = md.transposed != 0;
    const int cur = item_step<PH>(p, it) & 1;
    const int phase = item_phase<PH>(it);
    PhaseInfo pi;
    if (phase == kGram) {
        pi.a_mn = tr;
        pi.b_mn = tr;
        pi.mapA = xmap(maps, cur);
        pi.mapB = pi.mapA;
        pi.nkb = md.Qpad / C::BK;
    } else if (phase == kPoly) {
        pi.a_mn = false;
        pi.b_mn = false;
        pi.mapA = maps + 2 * 128;
        pi.mapB = pi.mapA;
        pi.nkb = md.Ppad / C::BK;
    } else {
        pi.a_mn = false;
        pi.b_mn = !tr;
        pi.mapA = maps + 3 * 128;
        pi.mapB = xmap(maps, cur);
        pi.nkb = md.Ppad / C::BK;
    }
    pi.mapAlo = pi.mapA;
    pi.mapBlo = pi.mapB;
    pi.nkr = pi.nkb;
    if constexpr (C::kSplit) {
        if (phase == kGram) {
            pi.mapAlo = xlo_map(maps, cur);
            pi.mapBlo = pi.mapAlo;
        } else if (phase == kPoly) {
            pi.mapAlo = maps + 7 * 128;
            pi.mapBlo = pi.mapAlo;
        } else {
            pi.mapAlo = maps + 6 * 128;
            pi.mapBlo = xlo_map(maps, cur);
        }
        pi.nkb = 3 * pi.nkr;
    }
    return pi;
}

// Main-loop K block kb of a tile: the operand maps it reads and its block kr
// of the product's K.  In bf16 hi/lo mode every product takes three products
// into one accumulator, A_hi B_hi + A_lo B_hi + A_hi B_lo (the product of the
// two low parts, 2^-16 relative, is left out), interleaved per K block: kb =
// 3 kr + pass, so that each K block's hi parts are read again while they are
// still in L2 (three whole passes over K in turn: Gram 7% slower on ViT-L/16
// and 560M shapes); otherwise one product.
struct KPass {
    const void* mapA;
    const void* mapB;
    int kr;
};
template <class C>
__device__ __forceinline__ KPass k_pass(const PhaseInfo& pi, int kb) {
    KPass k{pi.mapA, pi.mapB, kb};
    if constexpr (C::kSplit) {
        const int pass = kb % 3;
        k.kr = kb / 3;
        if (pass == 1)
            k.mapA = pi.mapAlo;
        else if (pass == 2)
            k.mapB = pi.mapBlo;
    }
    return k;
}

// A and M are stored only in the 256 x 256 tiles the Gram and the Poly
// compute (tile column >= tile row; no mirrored copy).  A product operand made
// of rows of A or M in tile row t reads K block kb (128 wide) K-major where it
// lies in a stored tile, and elsewhere MN-major from the stored transpose
// (rows kb, columns t), which equals it because A and M are symmetric: the
// Update's A operand (rows of M, t = tm) and both Poly operands (rows of A,
// t = tm and t = tn).  Both CTAs of a pair take the same choice.
__device__ __forceinline__ bool sym_mn(int kb, int t) { return (kb >> 1) < t; }

// The major-ness of a tile's A and B operand halves in K block kb: the
// phase's own choice (phase_info), or MN-major for rows of A or M outside
// the stored tiles.  The producer's copies and the MMA's descriptors use it.
template <int PH>
__device__ __forceinline__ bool a_mn_at(const PhaseInfo& pi, const GemmItem& it, int kb) {
    return pi.a_mn || (item_phase<PH>(it) != kGram && sym_mn(kb, it.tm));
}
template <int PH>
__device__ __forceinline__ bool b_mn_at(const PhaseInfo& pi, const GemmItem& it, int kb) {
    return pi.b_mn || (item_phase<PH>(it) == kPoly && sym_mn(kb, it.tn));
}

// Shared-memory descriptor of one K = 16 slice (kk) of a BK-wide K block:
// K-major: 128-byte rows (swizzle span), 8-row groups kKSbo apart, the K
// chunks of 64 elements one 128-row atom column (kAtomBytes) apart, slice kk
// 32 bytes further into its chunk; MN-major: 64-element MN chunks kMnLbo apart
// (LBO), 8-row K groups 1 KB apart (SBO), slice kk starts 16 rows = 2 KB
// further.
template <class C>
__device__ __forceinline__ uint64_t operand_desc(uint32_t base, int kk, bool mn) {
    return mn ? ptx::sdesc(base + kk * 16 * 128, C::kMnLbo, 1024, 2u)
              : ptx::sdesc(base + (kk >> 2) * C::kAtomBytes + (kk & 3) * 32, 16, C::kKSbo, C::kKLayout);
}

// Split K, one part of a tile: this warp stores its 32 rows of the part's
// fp32 accumulator (columns [32 ch_begin, 32 ch_end) of the tile, the share
// of epilogue warp group `group`) in the part's 256 x 256 slot, split_part +
// (sid + s) * 65536, column-major so that each column's 32 rows are one
// coalesced segment, and counts them in split_cnt[sid * 16 + rank * 8 +
// group * 4 + quad].  Returns true in the warp that counts last for its rows
// and columns (the other parts' values there are then visible to it); that
// warp resets the count for the next use.
__device__ __forceinline__ bool split_partial_is_last(const GemmLaunch& p, const GemmItem& it, int rank, int quad,
                                                      int group, int lane, uint32_t t_row, int ch_begin,
                                                      int ch_end) {
    const int parts = it.ksplit >> 8, own = it.ksplit & 0xff;
    const int row_t = rank * kBM + quad * 32 + lane;
    float* dst = p.split_part + (size_t(it.sid) + own) * 65536 + row_t;
    for (int ch = ch_begin; ch < ch_end; ++ch) {
        uint32_t r[32];
        ptx::tmem_ld_32x32b_x32(t_row + uint32_t(ch * 32), r);
        ptx::tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; ++j) dst[size_t(ch * 32 + j) * 256] = __uint_as_float(r[j]);
    }
    __threadfence();
    __syncwarp();
    uint32_t* cnt = p.split_cnt + size_t(it.sid) * 16 + rank * 8 + group * 4 + quad;
    int last = 0;
    if (lane == 0) {
        last = atomicAdd(cnt, 1u) == uint32_t(parts - 1) ? 1 : 0;
        if (last) *cnt = 0u;
    }
    last = __shfl_sync(0xffffffffu, last, 0);
    if (last) __threadfence();
    return last != 0;
}

// Staged epilogue stores (CTA-pair kernel).  A TMEM load gives each lane one
// row of a 32 x 32 chunk, so a lane's own 16-byte stores would touch 32 rows
// per instruction, half a 32-byte sector each.  Instead the warp stages the
// chunk in its own shared-memory buffer and stores it as 8 rows x 64 bytes per
// instruction, or transposed (column c of the chunk as a row of the output) as
// 8 columns x 64 bytes.  Rows are kStageRow bytes apart, so the 16-byte row
// writes of any 8 consecutive lanes fall in 8 different bank groups; each
// row's four 16-byte segments are rotated by row / 8, so that the column
// reads, which take 4 rows 8 apart per instruction (the same banks at any
// pitch that is a multiple of 16 bytes), fall in 4 different bank groups.
constexpr int kStageRow = 80;
constexpr int kStageWarpBytes = 32 * kStageRow;

// Row r's 16-byte segment q lies at r * kStageRow + 16 ((q + r / 8) mod 4).
__device__ __forceinline__ void stage_chunk(uint8_t* buf, int lane, const uint4 (&o)[4]) {
    uint8_t* row = buf + lane * kStageRow;
    const int rot = lane >> 3;
#pragma unroll
    for (int q = 0; q < 4; ++q) *reinterpret_cast<uint4*>(row + (((q + rot) & 3) << 4)) = o[q];
    __syncwarp();
}

// out[(r0 + r) * ld + c0 + c] = chunk[r][c]
__device__ __forceinline__ void put_rows(const uint8_t* buf, int lane, uint16_t* out, int64_t ld, int r0, int c0) {
    const int seg = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = i * 8 + (lane >> 2);
        const uint4 v = *reinterpret_cast<const uint4*>(buf + r * kStageRow + (((seg + i) & 3) << 4));  // r / 8 = i
        *reinterpret_cast<uint4*>(out + int64_t(r0 + r) * ld + c0 + seg * 8) = v;
    }
}

// out[(c0 + c) * ld + r0 + r] = chunk[r][c]
__device__ __forceinline__ void put_cols(const uint8_t* buf, int lane, uint16_t* out, int64_t ld, int r0, int c0) {
    const int seg = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int c = i * 8 + (lane >> 2);
        // rows seg * 8 .. + 7: rotated by seg
        const uint8_t* src = buf + (seg * 8) * kStageRow + ((c * 2 + (seg << 4)) & 63);
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const uint32_t lo = *reinterpret_cast<const uint16_t*>(src + (2 * e) * kStageRow);
            const uint32_t hi = *reinterpret_cast<const uint16_t*>(src + (2 * e + 1) * kStageRow);
            w[e] = lo | (hi << 16);
        }
        *reinterpret_cast<uint4*>(out + int64_t(c0 + c) * ld + r0 + seg * 8) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// The 32 x 32 chunk at src[(r0 + r) * ld + c0 + c] in the put_rows order:
// v[i] holds row 8 i + lane / 4, columns 8 (lane % 4) .. + 7.  The loads
// bypass L1 (the chunk was written by other SMs in the same launch).
__device__ __forceinline__ void get_rows(const uint16_t* src, int64_t ld, int r0, int c0, int lane, uint4 (&v)[4]) {
    const int seg = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i)
        v[i] = __ldcg(reinterpret_cast<const uint4*>(src + int64_t(r0 + i * 8 + (lane >> 2)) * ld + c0 + seg * 8));
}

// A chunk from get_rows, through the staging buffer, as this lane's row (in
// the buffer's plain layout, without the rotation: both of its accesses
// are row-wise and already spread over the bank groups).
__device__ __forceinline__ void own_row(uint8_t* buf, int lane, const uint4 (&v)[4], uint4 (&row)[4]) {
    const int seg = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) *reinterpret_cast<uint4*>(buf + (i * 8 + (lane >> 2)) * kStageRow + seg * 16) = v[i];
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 4; ++q) row[q] = *reinterpret_cast<const uint4*>(buf + lane * kStageRow + q * 16);
    __syncwarp();
}

// bf16 hi/lo mode: the low parts bf16(v - hi) of two values whose high parts
// are packed in hi.
__device__ __forceinline__ uint32_t lo_part2(float v0, float v1, uint32_t hi) {
    const float2 h = unpack2<true>(hi);
    return pack2<true>(v0 - h.x, v1 - h.y);
}

// Epilogue of one 128-row block of a finished tile: this warp's 32 TMEM lanes
// (rows row0 + 32 quad + [0, 32)) and the tile's 32-column chunks
// [ch_begin, ch_end) (chunk c: columns 256 tn + 32 c, TMEM columns t_row + 32 c).
//   Update: X' rows, stored in W's orientation (transposed iterates take one
//           coalesced 64-byte segment per column);
//   Gram / Poly: c * acc (+ b A + a I for Poly) into the Ppad x Ppad output,
//           the computed tile only (the skipped strictly-lower tiles are read
//           as the transpose of these, sym_mn).
// In the first step after the fused norm pass (p.fused_norm) the stored X_0
// is W itself: the Gram scales acc by x0_scale^2 and the Update by x0_scale.
// With split K (Gram), the accumulator is replaced by the sum, in part
// order, of the `parts` fp32 partials at split_tile (row row_t of the tile;
// this warp's own part among them).  STAGED: the stores go through the
// warp's staging buffer sbuf (kStageWarpBytes of shared memory).  SPLIT
// (bf16 hi/lo mode): the Gram and the Poly also store the low parts of A and
// M (the Poly's b A term reads both parts of A), and the Update those of X',
// except in the last step, which stores X_T in fp16 alone.
template <bool BF16, int PH, bool STAGED = false, bool SPLIT = false>
__device__ __forceinline__ void store_rows(const GemmLaunch& p, const GemmItem& it, const MatDev& md, int row0,
                                           uint32_t t_row, int quad, int lane, int ch_begin, int ch_end,
                                           const float* split_tile = nullptr, int parts = 1, int row_t = 0,
                                           uint8_t* sbuf = nullptr) {
    static_assert(BF16 || !SPLIT, "hi/lo parts are bf16");
    const int row_w = row0 + quad * 32;  // the warp's first row
    const int row = row_w + lane;
    const int nch = ch_end;
    const int t = item_step<PH>(p, it);
    const int phase = item_phase<PH>(it);
    const float xs = (p.fused_norm && t == 0) ? p.scalars[it.mat].x0_scale : 1.f;
    if (phase == kUpdate) {
        const int nb = (t & 1) ^ 1;
        uint16_t* out = reinterpret_cast<uint16_t*>(md.x[nb]);
        const bool f16_out = SPLIT && t == p.last_step;
        uint16_t* out_lo = (SPLIT && !f16_out) ? reinterpret_cast<uint16_t*>(md.xlo[nb]) : nullptr;
        const int64_t ld = md.ld;
        for (int ch = ch_begin; ch < nch; ++ch) {
            uint32_t r[32];
            ptx::tmem_ld_32x32b_x32(t_row + uint32_t(ch * 32), r);
            ptx::tmem_ld_wait();
            const int col0 = it.tn * kBNMax + ch * 32;
            uint4 o[4], l[4];
            uint32_t* ow = reinterpret_cast<uint32_t*>(o);
            uint32_t* lw = reinterpret_cast<uint32_t*>(l);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float v0 = xs * __uint_as_float(r[2 * j]), v1 = xs * __uint_as_float(r[2 * j + 1]);
                if (f16_out) {
                    ow[j] = pack2<false>(v0, v1);
                } else {
                    ow[j] = pack2<BF16>(v0, v1);
                    if (out_lo) lw[j] = lo_part2(v0, v1, ow[j]);
                }
            }
            if constexpr (STAGED) {
                // transposed iterates: X^T[q][p], the chunk's columns are rows of the buffer
                stage_chunk(sbuf, lane, o);
                if (md.transposed)
                    put_cols(sbuf, lane, out, ld, row_w, col0);
                else
                    put_rows(sbuf, lane, out, ld, row_w, col0);
                __syncwarp();
                if (out_lo) {
                    stage_chunk(sbuf, lane, l);
                    if (md.transposed)
                        put_cols(sbuf, lane, out_lo, ld, row_w, col0);
                    else
                        put_rows(sbuf, lane, out_lo, ld, row_w, col0);
                    __syncwarp();
                }
            } else if (md.transposed) {
                // X^T[q][p]: for each column the warp's 32 rows are contiguous
                const uint16_t* oh = reinterpret_cast<const uint16_t*>(o);
                uint16_t* dst = out + int64_t(col0) * ld + row;
#pragma unroll
                for (int j = 0; j < 32; ++j) dst[int64_t(j) * ld] = oh[j];
                if (out_lo) {
                    const uint16_t* lh = reinterpret_cast<const uint16_t*>(l);
                    uint16_t* dl = out_lo + int64_t(col0) * ld + row;
#pragma unroll
                    for (int j = 0; j < 32; ++j) dl[int64_t(j) * ld] = lh[j];
                }
            } else {
                uint4* dst = reinterpret_cast<uint4*>(out + int64_t(row) * ld + col0);
#pragma unroll
                for (int v = 0; v < 4; ++v) dst[v] = o[v];
                if (out_lo) {
                    uint4* dl = reinterpret_cast<uint4*>(out_lo + int64_t(row) * ld + col0);
#pragma unroll
                    for (int v = 0; v < 4; ++v) dl[v] = l[v];
                }
            }
        }
    } else {
        uint16_t* out = reinterpret_cast<uint16_t*>(phase == kGram ? md.a : md.b);
        const uint16_t* amat = reinterpret_cast<const uint16_t*>(md.a);
        const uint16_t* amat_lo = SPLIT ? reinterpret_cast<const uint16_t*>(md.alo) : nullptr;
        const int64_t ld = md.Ppad;
        const bool poly = phase == kPoly;
        uint16_t* out_lo = SPLIT ? reinterpret_cast<uint16_t*>(poly ? md.blo : md.alo) : nullptr;
        const float ca = poly ? p.coef[3 * t] : 0.f, cb = poly ? p.coef[3 * t + 1] : 0.f;
        const float cacc = poly ? p.coef[3 * t + 2] : xs * xs;
        // Poly reads b A at the output position: loads for the next chunk are
        // issued before the current chunk is processed (staged: coalesced
        // loads, turned into this lane's row through the staging buffer).  In
        // bf16 hi/lo mode the main loop, three products long, leaves the
        // epilogue time enough without the prefetch, and both parts are read.
        uint4 e_next[4];
        if (poly && !SPLIT) {
            if constexpr (STAGED) {
                get_rows(amat, ld, row_w, it.tn * kBNMax + ch_begin * 32, lane, e_next);
            } else {
                const uint4* src =
                    reinterpret_cast<const uint4*>(amat + int64_t(row) * ld + it.tn * kBNMax + ch_begin * 32);
#pragma unroll
                for (int q = 0; q < 4; ++q) e_next[q] = __ldcg(src + q);
            }
        }
        for (int ch = ch_begin; ch < nch; ++ch) {
            const int col0 = it.tn * kBNMax + ch * 32;
            const int64_t off = int64_t(row) * ld + col0;
            uint4 e[4], el[4];
            if (poly && SPLIT) {
                if constexpr (STAGED) {
                    uint4 v[4];
                    get_rows(amat, ld, row_w, col0, lane, v);
                    own_row(sbuf, lane, v, e);
                    get_rows(amat_lo, ld, row_w, col0, lane, v);
                    own_row(sbuf, lane, v, el);
                } else {
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        e[q] = __ldcg(reinterpret_cast<const uint4*>(amat + off) + q);
                        el[q] = __ldcg(reinterpret_cast<const uint4*>(amat_lo + off) + q);
                    }
                }
            } else if (poly) {
                if constexpr (STAGED) {
                    own_row(sbuf, lane, e_next, e);
                    if (ch + 1 < nch) get_rows(amat, ld, row_w, col0 + 32, lane, e_next);
                } else {
#pragma unroll
                    for (int q = 0; q < 4; ++q) e[q] = e_next[q];
                    if (ch + 1 < nch) {
                        const uint4* src = reinterpret_cast<const uint4*>(amat + off + 32);
#pragma unroll
                        for (int q = 0; q < 4; ++q) e_next[q] = __ldcg(src + q);
                    }
                }
            }
            uint32_t r[32];
            if (split_tile == nullptr) {
                ptx::tmem_ld_32x32b_x32(t_row + uint32_t(ch * 32), r);
                ptx::tmem_ld_wait();
            } else {
                // every part from memory, in part order: the sum does not
                // depend on which part finished last
                const float* src = split_tile + size_t(ch * 32) * 256 + row_t;
#pragma unroll
                for (int j = 0; j < 32; ++j) r[j] = __float_as_uint(__ldcg(src + size_t(j) * 256));
                for (int q = 1; q < parts; ++q) {
                    const float* s1 = src + size_t(q) * 65536;
                    float a[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) a[j] = __ldcg(s1 + size_t(j) * 256);
#pragma unroll
                    for (int j = 0; j < 32; ++j) r[j] = __float_as_uint(__uint_as_float(r[j]) + a[j]);
                }
            }
            uint4 o[4], l[4];
            uint32_t* ow = reinterpret_cast<uint32_t*>(o);
            uint32_t* lw = reinterpret_cast<uint32_t*>(l);
            const int d = row - col0;  // diagonal element of this row, if in the chunk
            const uint32_t* ew = reinterpret_cast<const uint32_t*>(e);
            const uint32_t* elw = reinterpret_cast<const uint32_t*>(el);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                float v0 = cacc * __uint_as_float(r[2 * j]);
                float v1 = cacc * __uint_as_float(r[2 * j + 1]);
                if (poly) {
                    // M = c A^2 + b A + a I
                    float2 x = unpack2<BF16>(ew[j]);
                    if (SPLIT) {
                        const float2 xl = unpack2<BF16>(elw[j]);
                        x.x += xl.x;
                        x.y += xl.y;
                    }
                    v0 = fmaf(cb, x.x, v0) + (2 * j == d ? ca : 0.f);
                    v1 = fmaf(cb, x.y, v1) + (2 * j + 1 == d ? ca : 0.f);
                }
                ow[j] = pack2<BF16>(v0, v1);
                if (out_lo) lw[j] = lo_part2(v0, v1, ow[j]);
            }
            // The output is symmetric and strictly-lower tiles are skipped,
            // with no mirrored copy: its readers take the missing blocks
            // MN-major from the stored ones (sym_mn).

            if constexpr (STAGED) {
                stage_chunk(sbuf, lane, o);
                put_rows(sbuf, lane, out, ld, row_w, col0);
                __syncwarp();
                if (out_lo) {
                    stage_chunk(sbuf, lane, l);
                    put_rows(sbuf, lane, out_lo, ld, row_w, col0);
                    __syncwarp();
                }
                continue;
            }
            uint4* dst = reinterpret_cast<uint4*>(out + off);
#pragma unroll
            for (int q = 0; q < 4; ++q) dst[q] = o[q];
            if (out_lo) {
                uint4* dl = reinterpret_cast<uint4*>(out_lo + off);
#pragma unroll
                for (int q = 0; q < 4; ++q) dl[q] = l[q];
            }
        }
    }
}

}  // namespace tc
}  // namespace slorr
