// milo_chunk.cu -- the chunk grid: the split-K decode with one thread block
// of four warps per chunk and row group of 8 query rows (8 of the batch x G
// rows of a KV head), or of two warps per row group and a pair of row groups
// once a KV head has more than 8 rows; three blocks per SM at head dimension
// 128.  Each chunk is streamed through two shared-memory slots that all the
// block's warps read.
//
// A chunk is a token range of one prefix entry (block b, KV head g).  Its
// block walks a fixed sequence of pieces, each at most kPieceBytes and
// brought by bulk copies into one of two slots while the warps work on the
// other:
//
//   P^K pieces   q~ = scale * log2(e) * P^K q for up to kPieceBytes / (2 d)
//                ranks per piece (Eq. 3 folded into Eq. 1), the 16-rank steps
//                dealt round-robin to the warps; q~ is kept as bf16 hi + lo
//                rows of the score A operand.
//   C pieces     whole 32-token tiles (C^K rows, then C^V rows of the same
//                tokens): scores s = C^K q~, an online softmax with a lazily
//                raised reference max, rank-space values v~ += C^V^T p.  Up
//                to 64 ranks the warps take whole tiles round-robin, above
//                that 16-token halves; each warp keeps its own softmax state.
//   P^V pieces   o += P^V^T v~ over up to kPieceBytes / (2 d) ranks per piece
//                (Alg. 1 Stage 2's back-projection), after the warps' v~ are
//                merged; each warp produces a share of the head dimension.
//
// A plan held as INT8 codes in device memory is read directly by a variant
// (Q8) that copies each piece's codes and group parameters and reads them
// back into bf16 cores in shared memory before the steps above.
//
// A dense-tail item (the tail of one query and KV head for the query's G
// rows, or 8 of them when G > 8: 1, or tail_pieces when the grid holds tails
// alone, pieces of kTailTokens tokens) brings each piece's K and V rows with 3-D TMA boxes (64 head
// dimensions x kTailTokens rows each, 128-byte rows with the 128-byte swizzle: few, wide requests)
// and runs the C steps on them with q~ = scale * log2(e) * q, a share of the
// tokens per warp; its values are already o.  Every item then adds its result
// into fp32 accumulators of its KV head's rows (see add_part) and exits; a
// small finish grid chained by programmatic dependent launch (one warp per KV
// head and row group) writes the normalised output.  No block waits on
// another.
//
// Shared-memory cores are 8 rows x 16 bytes (rows = tokens or ranks).  Every
// wait is bounded (~2 s) and sets MILO_ERR_TIMEOUT.
#include <cuda.h>
#include <cuda_bf16.h>

#include <type_traits>

#include "milo.h"
#include "milo_int8.cuh"
#include "milo_internal.h"
#include "milo_merge.cuh"
#include "milo_ptx.cuh"

namespace milo {
namespace {

constexpr int kPieceBytes = 32768;  // one slot
constexpr int kQ8Raw = 16384;       // reading an INT8 plan: one piece's codes (at most 256 cores)
constexpr int kTile = 32;           // tokens per tile
// warps per row group of 8 query rows: four when a block holds one row
// group (more warps in flight on each SM's three blocks), two when it holds
// two (their exchange areas share one slot)
template <int RG>
constexpr int kWarpsOf = RG == 1 ? 4 : 2;

// Shared memory of a block of RG row groups (RG x kWarpsOf<RG> warps).
template <int D, int RG>
struct CLay {
    static constexpr int kQ = 2 * kPieceBytes;                  // per row group: q~ (then v~) A fragments
    static constexpr int kQStride = (D / 16) * 32 * 16;         //   [D/16][32 lanes][4 words]
    static constexpr int kZero = kQ + RG * kQStride;            // a zero core line
    static constexpr int kBar = kZero + 128;                    // 2 mbarriers
    static constexpr int kX = kBar + 16;                        // per row group: m, l [kWarps][8], ref [8]
    static constexpr int kXStride = 16 * kWarpsOf<RG> + 8;      //   (words)
    static constexpr int kTotal = kX + (RG * kXStride * 4 + 15) / 16 * 16;
    // reading an INT8 plan: per slot, a piece's parameter words (at most 256
    // cores and 12 words of alignment)
    static constexpr int kPrm = kTotal;
    static constexpr int kPrmSlot = 1088;
    static constexpr int kTotalQ8 = kPrm + 2 * kPrmSlot;
    static constexpr int kRanksPerPiece = kPieceBytes / (D * 2);  // P^K / P^V rows per piece
};

// The pieces of a prefix chunk, in order: P^K, C, P^V.
struct Pieces {
    int npk, nc, npv;   // pieces of each kind
    int tpp;            // tiles per C piece
    int rpp;            // rank 8-groups per P piece
    __device__ int total() const { return npk + nc + npv; }
};

template <int D>
__device__ __forceinline__ Pieces pieces_of(const ChunkDev &c)
{
    Pieces s;
    s.rpp = CLay<D, 1>::kRanksPerPiece / 8;
    s.npk = (c.nrk + s.rpp - 1) / s.rpp;
    s.npv = (c.nrv + s.rpp - 1) / s.rpp;
    // an entry of rank 0 in K and V has no coefficient rows: its (at most
    // 32-token) chunk is one C piece that copies nothing
    const int row_bytes = kTile * (c.nrk + c.nrv) * 16;
    s.tpp = row_bytes > 0 ? max(1, kPieceBytes / row_bytes) : kChunkMaxTok / kTile;
    s.nc = (c.ntok + s.tpp * kTile - 1) / (s.tpp * kTile);
    return s;
}

// A piece of an INT8 plan read directly: up to two runs of consecutive cores
// (a C piece: the C^K rows, then the C^V rows).  Each run's 64-byte code
// groups land in the piece's raw slot, in order, and its parameter words in
// the slot's parameter area, copied in aligned groups of four (the run's
// first word at index core0 % 4 of its copy; run 1's copy follows run 0's).
struct Q8Piece {
    int64_t core0[2];  // first core of each run (packed byte offset / 128)
    int n[2];          // cores of each run
    int words[2];      // parameter words copied for each run (multiples of 4)
    int rg0, rlim;     // P pieces: first rank group, and the rank from which rows read back 0
};

template <int D>
__device__ __forceinline__ Q8Piece q8_piece(const ChunkDev &ch, const Pieces &ps, int k)
{
    Q8Piece q;
    q.core0[1] = 0;
    q.n[1] = 0;
    q.rg0 = 0;
    q.rlim = 1 << 30;  // C pieces: nothing to clear
    if (k < ps.npk) {
        const int r0 = k * ps.rpp, r1 = min(r0 + ps.rpp, ch.nrk);
        q.core0[0] = ch.pk / 128 + (int64_t)r0 * (D / 8);
        q.n[0] = (r1 - r0) * (D / 8);
        q.rg0 = r0;
        q.rlim = ch.rk;
    } else if (k < ps.npk + ps.nc) {
        const int t0 = (k - ps.npk) * ps.tpp * kTile;
        const int tg = (min(t0 + ps.tpp * kTile, ch.tok8) - t0) / 8;  // token groups
        q.core0[0] = ch.ck / 128 + (int64_t)(t0 / 8) * ch.nrk;
        q.n[0] = tg * ch.nrk;
        q.core0[1] = ch.cv / 128 + (int64_t)(t0 / 8) * ch.nrv;
        q.n[1] = tg * ch.nrv;
    } else {
        const int r0 = (k - ps.npk - ps.nc) * ps.rpp, r1 = min(r0 + ps.rpp, ch.nrv);
        q.core0[0] = ch.pv / 128 + (int64_t)r0 * (D / 8);
        q.n[0] = (r1 - r0) * (D / 8);
        q.rg0 = r0;
        q.rlim = ch.rv;
    }
#pragma unroll
    for (int j = 0; j < 2; ++j) q.words[j] = q.n[j] ? ((int)(q.core0[j] & 3) + q.n[j] + 3) & ~3 : 0;
    return q;
}

// KV head g, rows 8 rg .. 8 rg + 7, after every item: fold the listed
// records into the accumulators, write the output rows, clear the
// accumulators and the list.  Lane l: row 8 rg + l / 4, quarter l % 4 of the
// head dimension.
template <int D>
__device__ void finish_head(const DecodeParams &p, int g, int rg, int lane)
{
    const int gr = g * p.nrg + rg;  // this (KV head, row group)'s list
    const int64_t list_base = (int64_t)gr * p.list_cap;
    constexpr int kF4 = D / 16;  // float4 columns per quarter
    const int recf = 8 * D + kRecFloatsExtra;
    const int row = rg * 8 + (lane >> 2), qq = lane & 3;  // the KV head's query row (batch x heads)
    const int64_t ai = (int64_t)g * p.rows_max + row;
    float4 *Oq = reinterpret_cast<float4 *>(p.acc_o + ai * D + qq * (D / 4));
    const uint32_t mb = __ldcg(p.acc_m + ai);
    float M = mb ? ref_dec(mb) : -INFINITY;
    float Lsum = __ldcg(p.acc_l + ai);
    float4 acc[kF4];
#pragma unroll
    for (int f = 0; f < kF4; ++f) acc[f] = __ldcg(Oq + f);
    const uint32_t nov = __ldcg(p.ovf_cnt + gr);
#pragma unroll 1
    for (uint32_t k = 0; k < nov; ++k) {
        const int4 e = __ldcg(reinterpret_cast<const int4 *>(p.ovf_list) + list_base + k);
        const int rr = row - e.y;  // this row's row in the record
        if (rr < 0 || rr >= e.z) continue;
        const float *r = p.rec + (int64_t)e.x * recf;
        const float mr = __ldcg(r + 8 * D + rr), lr = __ldcg(r + 8 * D + 8 + rr);
        const float Mn = fmaxf(M, mr);
        const float a = exp2_diff(M, Mn), b = exp2_diff(mr, Mn);
        Lsum = Lsum * a + lr * b;
#pragma unroll
        for (int f = 0; f < kF4; ++f) {
            const float4 o = __ldcg(reinterpret_cast<const float4 *>(r + rr * D + qq * (D / 4)) + f);
            acc[f] = make_float4(acc[f].x * a + o.x * b, acc[f].y * a + o.y * b, acc[f].z * a + o.z * b,
                                 acc[f].w * a + o.w * b);
        }
        M = Mn;
    }
    if (row < p.rows_g) {
        const float inv = 1.f / Lsum;
        const int i = row / p.G, hh = row % p.G;
        float4 *dst = reinterpret_cast<float4 *>(p.out + ((int64_t)i * p.hq + g * p.G + hh) * D + qq * (D / 4));
#pragma unroll
        for (int f = 0; f < kF4; ++f)
            dst[f] = make_float4(acc[f].x * inv, acc[f].y * inv, acc[f].z * inv, acc[f].w * inv);
    }
    // clear for the next call
#pragma unroll
    for (int f = 0; f < kF4; ++f) __stcg(Oq + f, make_float4(0.f, 0.f, 0.f, 0.f));
    if (qq == 0) {
        __stcg(p.acc_l + ai, 0.f);
        __stcg(p.acc_m + ai, 0u);
    }
    if (lane == 0) __stcg(p.ovf_cnt + gr, 0u);
}

// This warp's share of an item's contribution to KV head g: head-dimension
// columns 8 (n0 + n) + 2 c4, + 1 of row r4 (ov[n]), for rows arow = row0 + r4
// with r4 < nrows.  M is the item's row maximum, lsum its row sum (used when
// with_l), refb the row's reference (encoded; 0 = unset).  Returns whether the
// item went to the accumulators (the same in every warp of the row group:
// their inputs agree);
// otherwise the warp wrote its columns of the item's record.
template <int D, int NC>
__device__ bool add_part(const DecodeParams &p, int g, int lane, int n0, const float (&ov)[NC][2], float M,
                         float lsum, uint32_t refb, bool with_l, int row0, int nrows, int64_t rec_idx)
{
    const int r4 = lane >> 2, c4 = lane & 3;
    const bool row_ok = r4 < nrows;
    const float Mref = refb ? ref_dec(refb) : M;  // unset only when the row saw no token
    const bool direct = __all_sync(0xffffffffu, !row_ok || !(M - Mref > kDirectMax));
    if (direct) {
        if (row_ok && M != -INFINITY) {
            const float f = ex2_approx(M - Mref);
            float *orow = p.acc_o + ((int64_t)g * p.rows_max + row0 + r4) * D + 8 * n0 + 2 * c4;
#pragma unroll
            for (int n = 0; n < NC; ++n)
                atomicAdd(reinterpret_cast<float2 *>(orow + 8 * n), make_float2(f * ov[n][0], f * ov[n][1]));
            if (with_l && c4 == 0) atomicAdd(p.acc_l + (int64_t)g * p.rows_max + row0 + r4, f * lsum);
        }
    } else {
        // an outlier maximum: the item keeps a record for the final merge
        float *rec = p.rec + rec_idx * (8 * D + kRecFloatsExtra);
#pragma unroll
        for (int n = 0; n < NC; ++n)
            __stcg(reinterpret_cast<float2 *>(rec + r4 * D + 8 * (n0 + n) + 2 * c4), make_float2(ov[n][0], ov[n][1]));
        if (with_l && c4 == 0) {
            __stcg(rec + 8 * D + r4, M);
            __stcg(rec + 8 * D + 8 + r4, lsum);
        }
    }
    return direct;
}

// RG row groups of 8 query rows per block, kWarpsOf<RG> warps each: the groups
// share every piece (RG = 2 for calls with several row groups per KV head).
// A tail block holds RG tail items, one per group; with RG = 2 group i's
// item sits in slot i, with RG = 1 its pieces alternate between the slots.  "warp" below is the
// warp's index within its row group.  Q8: the plan is held as INT8 codes,
// read directly (p.q8_codes, p.q8_params).
template <int D, int RG, bool Q8>
__global__ void __launch_bounds__(32 * kWarpsOf<RG> * RG, 3)
    chunk_kernel(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tmap_k,
                 const __grid_constant__ CUtensorMap tmap_v)
{
    static_assert(RG == 1 || RG == 2, "one or two row groups per block");
    static_assert(2 * (D / 8) * kTailTokens * 16 <= (RG == 1 ? 2 : 1) * kPieceBytes,
                  "a group's tail item fits its slots");
    using L = CLay<D, RG>;
    constexpr int kWarps = kWarpsOf<RG>;
    constexpr int kThreads = 32 * kWarps * RG;
    constexpr int KD = D / 16;  // 16-wide k-steps over the head dimension
    constexpr int NT = D / 8;   // 8-wide tiles over the head dimension (and the largest rank)
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, lane = tid & 31;
    // row group of the block, warp in it
    const int grp = RG == 1 ? 0 : (tid >> 5) / kWarps, warp = RG == 1 ? tid >> 5 : (tid >> 5) % kWarps;
    const int r4 = lane >> 2, c4 = lane & 3;  // mma fragment row and column pair
    const int mi = lane >> 3, mr = lane & 7;  // ldmatrix: matrix and row this lane addresses
    uint4 *sq = reinterpret_cast<uint4 *>(smem + L::kQ + grp * L::kQStride);
    float *sx_m = reinterpret_cast<float *>(smem + L::kX) + grp * L::kXStride;  // [warp][row]
    float *sx_l = sx_m + 8 * kWarps;                             // [warp][row]
    uint32_t *sx_ref = reinterpret_cast<uint32_t *>(sx_l + 8 * kWarps);  // [row]
    const uint32_t zline = smem_u32(smem + L::kZero) + mr * 16;
    const uint32_t bar0 = smem_u32(smem + L::kBar);
    // blocks [0, num_chunks * nrgb): chunk blockIdx / nrgb for row groups
    // RG (blockIdx % nrgb) + grp (the blocks of one chunk are neighbours, so
    // they read its pieces from L2); then the dense-tail items, RG a block
    const int nrgb = (p.nrg + RG - 1) / RG;
    const int nprefix = p.num_chunks * nrgb;
    const bool is_tail = (int)blockIdx.x >= nprefix;
    const int rgrp = is_tail ? 0 : ((int)blockIdx.x % nrgb) * RG + grp;
    const int item = is_tail ? ((int)blockIdx.x - nprefix) * RG + grp : 0;
    // a group past the last row group or tail item only keeps the barriers
    // (with one group per block there is none)
    const bool active = RG == 1 || (is_tail ? item < p.num_tail_items : rgrp < p.nrg);

    pdl_trigger();
    // zero the slots, q~ and the zero line: reads past a piece's data then
    // see finite values (the copies below are ordered after these stores).
    // A tail block reads only the rows its boxes write (out-of-range rows
    // arrive as zeros) and no rank padding, so its slots stay as they are.
    for (int i = tid + (is_tail ? L::kQ / 16 : 0); i < L::kBar / 16; i += kThreads)
        reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");

    ChunkDev ch = {};
    Pieces ps = {};
    int g = 0, ntok = 0, nrk = 0, nrv = 0;
    if (!is_tail) {
        ch = p.chunks[blockIdx.x / nrgb];
        ps = pieces_of<D>(ch);
        g = ch.g;
        ntok = ch.ntok;
        nrk = ch.nrk;
        nrv = ch.nrv;
    }
    // piece k into slot k & 1 (thread 0)
    auto issue = [&](int k) {
        const uint32_t bar = bar0 + 8 * (k & 1), dst = smem_u32(smem) + (k & 1) * kPieceBytes;
        if constexpr (Q8) {
            // an INT8 plan: codes in raw slot k & 1, parameters in its parameter area
            const Q8Piece q = q8_piece<D>(ch, ps, k);
            const uint32_t cdst = smem_u32(smem) + (k & 1) * kQ8Raw;
            const uint32_t pdst = smem_u32(smem) + L::kPrm + (k & 1) * L::kPrmSlot;
            mbar_arrive_tx(bar, 64u * (uint32_t)(q.n[0] + q.n[1]) + 4u * (uint32_t)(q.words[0] + q.words[1]));
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                if (q.n[j] == 0) continue;
                bulk_g2s(cdst + (j ? 64u * q.n[0] : 0u), p.q8_codes + q.core0[j] * 64, 64u * q.n[j], bar);
                bulk_g2s(pdst + (j ? 4u * q.words[0] : 0u), p.q8_params + (q.core0[j] & ~(int64_t)3),
                         4u * q.words[j], bar);
            }
            return;
        }
        if (k < ps.npk) {
            const int r0 = k * ps.rpp, r1 = min(r0 + ps.rpp, ch.nrk);
            const uint32_t b = (uint32_t)(r1 - r0) * D * 16;
            mbar_arrive_tx(bar, b);
            bulk_g2s(dst, p.packed + ch.pk + (int64_t)r0 * D * 16, b, bar);
        } else if (k < ps.npk + ps.nc) {
            const int t0 = (k - ps.npk) * ps.tpp * kTile;
            const int r8 = min(t0 + ps.tpp * kTile, ch.tok8) - t0;  // rows (a multiple of 8)
            const uint32_t kb = (uint32_t)r8 * ch.nrk * 16, vb = (uint32_t)r8 * ch.nrv * 16;
            // (a side of rank 0 copies nothing; with both, the arrival alone
            // completes the phase)
            mbar_arrive_tx(bar, kb + vb);
            if (kb) bulk_g2s(dst, p.packed + ch.ck + (int64_t)t0 * ch.nrk * 16, kb, bar);
            if (vb) bulk_g2s(dst + kb, p.packed + ch.cv + (int64_t)t0 * ch.nrv * 16, vb, bar);
        } else {
            const int r0 = (k - ps.npk - ps.nc) * ps.rpp, r1 = min(r0 + ps.rpp, ch.nrv);
            const uint32_t b = (uint32_t)(r1 - r0) * D * 16;
            mbar_arrive_tx(bar, b);
            bulk_g2s(dst, p.packed + ch.pv + (int64_t)r0 * D * 16, b, bar);
        }
    };
    if (tid == 0) {
        mbar_init(bar0, 1);
        mbar_init(bar0 + 8, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (!is_tail) {
            issue(0);
            if (ps.total() > 1) issue(1);
        }
    }
    // warm L2 with the group's q rows, the first load after the wait (a
    // prefetch reads nothing into the block, so it may precede the wait)
    if (warp == 0 && lane < 16 && active) {
        const int r = lane >> 1;
        int qrow = -1, gq = g;
        if (is_tail) {
            const int rq = (item / p.tail_splits) % p.nrg_t;
            gq = (item / (p.tail_splits * p.nrg_t)) % p.hkv;
            if (8 * rq + r < p.G) qrow = item / (p.hkv * p.tail_splits * p.nrg_t) * p.G + 8 * rq + r;
        } else if (8 * rgrp + r < p.rows_g) {
            qrow = 8 * rgrp + r;
        }
        if (qrow >= 0)
            prefetch_l2(p.q + ((int64_t)(qrow / p.G) * p.hq + gq * p.G + qrow % p.G) * D + (lane & 1) * (D / 2));
    }
    __syncthreads();
    pdl_wait();  // q, the tails and the accumulators belong to the preceding grids until here

    // the warp's online-softmax state and rank-space values
    float m_w = -INFINITY, l_w = 0.f;
    float vacc[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n) vacc[n][0] = vacc[n][1] = vacc[n][2] = vacc[n][3] = 0.f;

    // One tile of TT (16 or 32) tokens at token tb of the tile data: C^K core
    // (tg, rg) at kb + tg * ktg + rg * KRG, C^V core at vb + tg * vtg + rg * VRG
    // (SWZ: a dense-tail item, whose core (tg, cg) row r lies in TMA box
    // cg / 8 at row 8 tg + r, 16-byte chunk (cg % 8) ^ r, boxes KRG apart);
    // tg8 token groups present, tokens < nv valid, at least one of them in
    // this tile.  R16 (at least both ranks / 16) fixes the 16-rank steps;
    // R16, TT, KRG and VRG are compile-time constants, so that the body is one
    // straight block whose loads take immediate offsets.  Token groups past
    // the data read the last one (their scores are masked and their p is 0).
    // Rank groups past a rank read whatever follows in shared memory (finite:
    // the slots are zeroed at start, and the furthest such read ends inside
    // the q~ area): for scores their q~ is 0, and the rank-space values they
    // give are never back-projected.
    auto tile = [&](auto r16c, auto ttc, auto krgc, auto vrgc, auto swzc, uint32_t kb, uint32_t ktg, uint32_t vb,
                    uint32_t vtg, int tb, int tg8, int nv) {
        constexpr int R16 = decltype(r16c)::value;
        constexpr int NH = decltype(ttc)::value / 16;  // 16-token halves
        constexpr uint32_t KRG = decltype(krgc)::value, VRG = decltype(vrgc)::value;
        constexpr bool SWZ = decltype(swzc)::value;
        // per half h: this lane's ldmatrix row address at rank step 0
        uint32_t kh[NH], vh[NH];
        // swizzled: the 16-byte chunk of column group 2k + b in row r is
        // (2 (k % 4) ^ (r & 6)) | ((b ^ r) & 1): the first part per k % 4
        uint32_t sw[4] = {0u, 0u, 0u, 0u};
        if constexpr (SWZ) {
#pragma unroll
            for (int j = 0; j < 4; ++j) sw[j] = (uint32_t)((2 * j) ^ (mr & 6)) << 4;
        }
#pragma unroll
        for (int h = 0; h < NH; ++h) {
            // scores, matrices (tg0, 2ks), (tg0, 2ks + 1), (tg0 + 1, 2ks), (tg0 + 1, 2ks + 1)
            const int tgk = min(tb / 8 + 2 * h + (mi >> 1), tg8 - 1);
            // values (transposed), matrices (tg0, 2jp), (tg0 + 1, 2jp), (tg0, 2jp + 1), (tg0 + 1, 2jp + 1)
            const int tgv = min(tb / 8 + 2 * h + (mi & 1), tg8 - 1);
            if constexpr (SWZ) {
                kh[h] = kb + tgk * 1024 + mr * 128 + ((((mi & 1) ^ mr) & 1) << 4);
                vh[h] = vb + tgv * 1024 + mr * 128 + ((((mi >> 1) ^ mr) & 1) << 4);
            } else {
                kh[h] = kb + tgk * ktg + (mi & 1) * KRG + mr * 16;
                vh[h] = vb + tgv * vtg + (mi >> 1) * VRG + mr * 16;
            }
        }
        float s4[2 * NH][4];
#pragma unroll
        for (int n = 0; n < 2 * NH; ++n) s4[n][0] = s4[n][1] = s4[n][2] = s4[n][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < R16; ++ks) {
            const uint4 q4 = sq[ks * 32 + lane];
            const uint32_t qa[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4(SWZ ? kh[h] + (ks >> 2) * KRG + sw[ks & 3] : kh[h] + 2 * ks * KRG, b0, b1, b2, b3);
                mma16816(s4[2 * h], qa, b0, b1);
                mma16816(s4[2 * h + 1], qa, b2, b3);
            }
        }
        // score of token tb + 8n + 2 c4 + j: hi rows + lo rows
        const int nl = nv - tb - 2 * c4;  // this lane's tokens 8n + j are valid while 8n + j < nl
        float sv[4 * NH];
#pragma unroll
        for (int n = 0; n < 2 * NH; ++n) {
            sv[2 * n] = 8 * n < nl ? s4[n][0] + s4[n][2] : -INFINITY;
            sv[2 * n + 1] = 8 * n + 1 < nl ? s4[n][1] + s4[n][3] : -INFINITY;
        }
        float lm[4 * NH];
#pragma unroll
        for (int j = 0; j < 4 * NH; ++j) lm[j] = sv[j];
#pragma unroll
        for (int w = 2 * NH; w >= 1; w /= 2)
#pragma unroll
            for (int j = 0; j < w; ++j) lm[j] = fmaxf(lm[j], lm[j + w]);
        // lazy rescale (p stays <= 2^8): the row maximum is formed only when
        // some score passes the reference by more than 8.  Every row has a
        // valid score in the warp's first tile, so m_w is finite from then on.
        if (__any_sync(0xffffffffu, lm[0] > m_w + 8.f)) {
            const float mx = quad_max(lm[0]);
            if (mx > m_w + 8.f) {
                const float alpha = exp2_diff(m_w, mx);
                l_w *= alpha;
#pragma unroll
                for (int n = 0; n < NT; ++n) {
                    vacc[n][0] *= alpha;
                    vacc[n][1] *= alpha;
                    vacc[n][2] *= alpha;
                    vacc[n][3] *= alpha;
                }
                m_w = mx;
            }
        }
        float pr[4 * NH];
#pragma unroll
        for (int j = 0; j < 4 * NH; ++j) pr[j] = ex2_approx(sv[j] - m_w);  // a masked score gives 0
        float ls[4 * NH];
#pragma unroll
        for (int j = 0; j < 4 * NH; ++j) ls[j] = pr[j];
#pragma unroll
        for (int w = 2 * NH; w >= 1; w /= 2)
#pragma unroll
            for (int j = 0; j < w; ++j) ls[j] += ls[j + w];
        l_w += ls[0];
        // A fragments of p for the 16-token halves (rows 0-7 hi, 8-15 lo)
        uint32_t pa[NH][4];
#pragma unroll
        for (int h = 0; h < NH; ++h) {
            split_hi_lo(pr[4 * h], pr[4 * h + 1], pa[h][0], pa[h][1]);
            split_hi_lo(pr[4 * h + 2], pr[4 * h + 3], pa[h][2], pa[h][3]);
        }
#pragma unroll
        for (int jp = 0; jp < R16; ++jp) {
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(SWZ ? vh[h] + (jp >> 2) * VRG + sw[jp & 3] : vh[h] + 2 * jp * VRG, b0, b1, b2, b3);
                mma16816(vacc[2 * jp], pa[h], b0, b1);
                mma16816(vacc[2 * jp + 1], pa[h], b2, b3);
            }
        }
    };
    // f(integral_constant<int, v>) for v the least of 1, 2, 4, 8 that is >= n
    // (at most N): few variants, so that the instruction cache holds them
    auto dispatch = [&](auto nc, int n, auto &&f) {
        using std::integral_constant;
        constexpr int N = decltype(nc)::value;
        static_assert(N == 4 || N == 8, "4 or 8 cases");
        if (n <= 1) {
            f(integral_constant<int, 1>{});
        } else if (n <= 2) {
            f(integral_constant<int, 2>{});
        } else if (n <= 4 || N == 4) {
            f(integral_constant<int, 4>{});
        } else {
            f(integral_constant<int, N>{});
        }
    };

    const int np = ps.total();
    // Reading an INT8 plan (Q8), shared memory holds two raw slots of
    // kQ8Raw bytes at the start (the codes of pieces k & 1) and one bf16
    // slot after them, where each piece becomes the bf16 cores the bf16
    // piece would be (every thread): core i at byte 128 i, its values read
    // back as the staging kernel reads them (milo_int8.cuh), P rows past the
    // rank set to 0 (C padding stays as read back: it meets q~ = 0 or p = 0
    // only).  Eight neighbouring threads take the eight rows of a core (8
    // code bytes in, 16 bytes out: no bank conflicts).  The raw slot is free
    // again once the piece is read back, so piece k + 2 is requested then,
    // before the tiles run.  A tile's reads past the values (at most 2 KB)
    // land in the q~ area that follows the bf16 slot.
    auto q8_read = [&](int k) {
        const Q8Piece q = q8_piece<D>(ch, ps, k);
        const int n = q.n[0] + q.n[1];
        const uint8_t *raw = smem + (k & 1) * kQ8Raw;
        uint8_t *vals = smem + kPieceBytes;
        const uint32_t *prm = reinterpret_cast<const uint32_t *>(smem + L::kPrm + (k & 1) * L::kPrmSlot);
        const int pa = (int)(q.core0[0] & 3), pb = q.words[0] + (int)(q.core0[1] & 3) - q.n[0];
        const int row = tid & 7;
#pragma unroll 4
        for (int i = tid >> 3; i < n; i += kThreads / 8) {
            const uint2 c = *reinterpret_cast<const uint2 *>(raw + 64 * i + 8 * row);
            uint4 v = dequant_row(c, prm[i < q.n[0] ? pa + i : pb + i]);
            // P pieces: rank 8 (rg0 + i / (D / 8)) + row
            if (8 * (q.rg0 + i / (D / 8)) + row >= q.rlim) v = make_uint4(0u, 0u, 0u, 0u);
            *reinterpret_cast<uint4 *>(vals + 128 * i + 16 * row) = v;
        }
        // the raw slot's reads before its next copy (async proxy), the values
        // before the tiles
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (tid == 0 && k + 2 < np) issue(k + 2);
    };
    // wait for piece k (every warp); afterwards release its slot and bring
    // piece k + 2 into it
    auto wait_piece = [&](int k) {
        mbar_wait(bar0 + 8 * (k & 1), (k >> 1) & 1, p.status);
        if constexpr (Q8) {
            q8_read(k);
            return smem_u32(smem) + (uint32_t)kPieceBytes;
        }
        return smem_u32(smem) + (k & 1) * kPieceBytes;
    };
    auto release_piece = [&](int k) {
        if constexpr (Q8) {
            __syncthreads();  // the bf16 slot's reads before the next read-back
            return;
        }
        // the slot's reads are ordered before the async-proxy write
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (tid == 0 && k + 2 < np) issue(k + 2);
    };

    uint32_t ref = 0u;  // this row's reference maximum (warp 0, lane c4 == 0), see publish_ref
    int qi = 0, rq = 0;  // tail item: query, and group of 8 of its G heads
    const bool leader = RG == 1 ? tid == 0 : warp == 0 && lane == 0;  // the group's first thread
    if (is_tail) {
        // tail item: query qi, KV head g, tokens [t0, t0 + ntok) of qi's dense
        // tail in pieces of kTailTokens.  With one group a block (RG = 1) an
        // item holds up to p.tail_pieces pieces, streamed through the two
        // slots (piece k in slot k & 1, requested when piece k - 2 is
        // consumed); with two groups each group's item is one piece in the
        // group's slot.
        const int S = p.tail_splits, P = RG == 1 ? p.tail_pieces : 1;
        int64_t o0 = 0;
        int T = 0, sp = 0;
        if (active) {
            // item = ((qi * Hkv + g) * nrg_t + rq) * S + sp: rows [8 rq, 8 rq + 8) of qi's G heads
            sp = item % S;
            rq = (item / S) % p.nrg_t;
            g = (item / (S * p.nrg_t)) % p.hkv;
            qi = item / (S * p.nrg_t * p.hkv);
            o0 = p.tail_offsets[qi];
            T = (int)(p.tail_offsets[qi + 1] - o0);
        }
        if (sp == S - 1 && T > S * P * kTailTokens && leader)
            atomicCAS(p.status, 0, (int32_t)MILO_ERR_DEVICE_BOUNDS);
        const int t0 = sp * P * kTailTokens;
        ntok = max(0, min(t0 + P * kTailTokens, T) - t0);
        const int npieces = (ntok + kTailTokens - 1) / kTailTokens;
        nrk = nrv = NT;
        // K then V: one box of kTailTokens rows x 64 columns (128-byte rows,
        // 128-byte swizzle) per 64 columns; a box starts on a 1024-byte line
        constexpr uint32_t kBox = kTailTokens * 128, kHalf = (D / 64) * kBox;
        static_assert(kPieceBytes % 1024 == 0 && kHalf % 1024 == 0, "swizzled boxes on 1024-byte lines");
        auto tslot = [&](int k) { return (uint32_t)(RG == 1 ? (k & 1) : grp); };
        if (npieces > 0 && (smem_u32(smem) & 1023u)) {
            // (cannot happen: the dynamic shared memory starts on a 1024-byte
            // line) the item is dropped and the call reports a bounds error
            if (leader) atomicCAS(p.status, 0, (int32_t)MILO_ERR_DEVICE_BOUNDS);
            ntok = 0;
        }
        const int np_t = ntok > 0 ? npieces : 0;
        auto tail_issue = [&](int k) {
            const uint32_t base = smem_u32(smem) + tslot(k) * kPieceBytes, b = bar0 + 8 * tslot(k);
            mbar_arrive_tx(b, 2 * kHalf);
#pragma unroll
            for (int c = 0; c < D / 64; ++c) {
                tma_load_3d(base + c * kBox, &tmap_k, 64 * c, g, (int)(o0 + t0 + k * kTailTokens), b);
                tma_load_3d(base + kHalf + c * kBox, &tmap_v, 64 * c, g, (int)(o0 + t0 + k * kTailTokens), b);
            }
        };
        if (leader) {
            if (np_t > 0) tail_issue(0);
            if (np_t > 1) tail_issue(1);
        }
        // q~ = scale * log2(e) * q of the G heads of query qi, as score A fragments
        // (k-steps split between the warps)
#pragma unroll 1
        for (int ks = warp; ks < KD; ks += kWarps) {
            float x[4] = {0.f, 0.f, 0.f, 0.f};
            if (8 * rq + r4 < p.G) {
                const uint16_t *qr = p.q + ((int64_t)qi * p.hq + g * p.G + 8 * rq + r4) * D + 16 * ks + 2 * c4;
                const __nv_bfloat162 a2 = *reinterpret_cast<const __nv_bfloat162 *>(qr);
                const __nv_bfloat162 b2 = *reinterpret_cast<const __nv_bfloat162 *>(qr + 8);
                x[0] = __low2float(a2) * p.scale_log2;
                x[1] = __high2float(a2) * p.scale_log2;
                x[2] = __low2float(b2) * p.scale_log2;
                x[3] = __high2float(b2) * p.scale_log2;
            }
            uint4 f;
            split_hi_lo(x[0], x[1], f.x, f.y);
            split_hi_lo(x[2], x[3], f.z, f.w);
            sq[ks * 32 + lane] = f;
        }
        __syncthreads();
        // each piece's tokens in units of kTailTokens / kWarps, one per warp
        constexpr int kTU = kTailTokens / kWarps;
        static_assert(kTU == 16 || kTU == 32, "tail units of 16 or 32 tokens");
        const int tb = kTU * warp;
#pragma unroll 1
        for (int k = 0; k < np_t; ++k) {
            const uint32_t base = smem_u32(smem) + tslot(k) * kPieceBytes;
            mbar_wait(bar0 + 8 * tslot(k), (k >> 1) & 1, p.status);
            const int nk = min(kTailTokens, ntok - k * kTailTokens);
            if (tb < nk) {
                tile(std::integral_constant<int, NT / 2>{}, std::integral_constant<int, kTU>{},
                     std::integral_constant<uint32_t, kBox>{}, std::integral_constant<uint32_t, kBox>{},
                     std::true_type{}, base, 1024, base + kHalf, 1024, tb, kTailTokens / 8, nk);
                if (k == 0 && warp == 0)
                    ref = publish_ref(p, g, qi * p.G + 8 * rq + r4, 8 * rq + r4 < p.G, c4, m_w);
            }
            if (k + 2 < np_t) {
                // (RG = 1 here: P > 1) the slot's reads before its next copy
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncthreads();
                if (leader) tail_issue(k + 2);
            }
        }
    } else {
        // P^K pieces (the loops over the piece kinds keep each kind's
        // registers local to its loop)
        {
            // q rows of KV head g as the projection's B fragments (q^T)
            uint32_t qa[KD][2];
            const int qrow = 8 * rgrp + r4;  // the KV head's query row (batch x heads)
            const bool row_ok = qrow < p.rows_g;
            const uint16_t *qr = p.q + ((int64_t)(qrow / p.G) * p.hq + g * p.G + qrow % p.G) * D + 2 * c4;
#pragma unroll
            for (int ks = 0; ks < KD; ++ks) {
                qa[ks][0] = row_ok ? *reinterpret_cast<const uint32_t *>(qr + 16 * ks) : 0u;
                qa[ks][1] = row_ok ? *reinterpret_cast<const uint32_t *>(qr + 16 * ks + 8) : 0u;
            }
#pragma unroll 1
            for (int k = 0; k < ps.npk; ++k) {
                const uint32_t slot = wait_piece(k);
                // q~ for the 16-rank steps j of rank groups [r0, r1), j of this
                // warp's parity: A = P^K (16 ranks x 16 columns, cores (rg - r0,
                // cg) of this piece), B = q^T, so that one product covers 16
                // ranks; the accumulator [rank][row] is split into bf16 hi + lo
                // and transposed (movmatrix) into the score A layout.
                const int r0 = k * ps.rpp, r1 = min(r0 + ps.rpp, nrk);
                // (a piece never holds more 16-rank steps than q~ has: ranks <= D)
                constexpr int kNKMax = L::kRanksPerPiece / 16 < KD ? L::kRanksPerPiece / 16 : KD;
                if (active) dispatch(std::integral_constant<int, kNKMax>{}, (r1 - r0 + 1) / 2, [&](auto nkc) {
                    constexpr int NJ = (decltype(nkc)::value + kWarps - 1) / kWarps;  // steps per warp
                    float acc[NJ][2][4];
#pragma unroll
                    for (int jj = 0; jj < NJ; ++jj)
#pragma unroll
                        for (int e = 0; e < 4; ++e) acc[jj][0][e] = acc[jj][1][e] = 0.f;
#pragma unroll
                    for (int ks = 0; ks < KD; ++ks) {
#pragma unroll
                        for (int jj = 0; jj < NJ; ++jj) {
                            // matrices: (2j, 2ks), (2j + 1, 2ks), (2j, 2ks + 1), (2j + 1, 2ks + 1)
                            const int rl = 2 * (kWarps * jj + warp) + (mi & 1);
                            const uint32_t addr =
                                r0 + rl < r1 ? slot + (rl * NT + 2 * ks + (mi >> 1)) * 128 + mr * 16 : zline;
                            uint32_t a[4];
                            ldsm_x4(addr, a[0], a[1], a[2], a[3]);
                            mma16816(acc[jj][ks & 1], a, qa[ks][0], qa[ks][1]);
                        }
                    }
#pragma unroll
                    for (int jj = 0; jj < NJ; ++jj) {
                        // acc: ranks 16 j + r4 (regs 0, 1) and + 8 (regs 2, 3) for rows 2 c4, 2 c4 + 1
                        const int j = r0 / 2 + kWarps * jj + warp;
                        uint32_t hi0, lo0, hi1, lo1;
                        split_hi_lo((acc[jj][0][0] + acc[jj][1][0]) * p.scale_log2,
                                    (acc[jj][0][1] + acc[jj][1][1]) * p.scale_log2, hi0, lo0);
                        split_hi_lo((acc[jj][0][2] + acc[jj][1][2]) * p.scale_log2,
                                    (acc[jj][0][3] + acc[jj][1][3]) * p.scale_log2, hi1, lo1);
                        if (2 * j < r1 && j < KD)
                            sq[j * 32 + lane] = make_uint4(movm_t(hi0), movm_t(lo0), movm_t(hi1), movm_t(lo1));
                    }
                });
                release_piece(k);
            }
        }
        const int r16 = (max(nrk, nrv) + 1) / 2;
#pragma unroll 1
        for (int k = ps.npk; k < ps.npk + ps.nc; ++k) {
            const uint32_t slot = wait_piece(k);
            const int t0 = (k - ps.npk) * ps.tpp * kTile;
            const int nv = min(ps.tpp * kTile, ntok - t0);  // valid tokens of this piece
            const int r8 = min(t0 + ps.tpp * kTile, ch.tok8) - t0;
            const uint32_t vb = slot + (uint32_t)r8 * nrk * 16;
            if (active) dispatch(std::integral_constant<int, NT / 2>{}, r16, [&](auto r16c) {
                using std::integral_constant;
                if constexpr (decltype(r16c)::value <= 4) {
                    // up to 64 ranks: whole tiles round-robin over the warps
#pragma unroll 1
                    for (int tb = kTile * warp; tb < nv; tb += kWarps * kTile)
                        tile(r16c, integral_constant<int, kTile>{}, integral_constant<uint32_t, 128>{},
                             integral_constant<uint32_t, 128>{}, std::false_type{}, slot, nrk * 128, vb, nrv * 128,
                             tb, r8 / 8, nv);
                } else {
                    // above: 16-token halves of the tiles round-robin over the warps
#pragma unroll 1
                    for (int tb = 16 * warp; tb < nv; tb += kWarps * 16)
                        tile(r16c, integral_constant<int, 16>{}, integral_constant<uint32_t, 128>{},
                             integral_constant<uint32_t, 128>{}, std::false_type{}, slot, nrk * 128, vb, nrv * 128,
                             tb, r8 / 8, nv);
                }
            });
            if (k == ps.npk && warp == 0) ref = publish_ref(p, g, 8 * rgrp + r4, 8 * rgrp + r4 < p.rows_g, c4, m_w);
            release_piece(k);
        }
    }

    // ---- merge the warps' softmax states: M = max over the warps per row
    {
        const float lq = quad_sum(l_w);
        if (c4 == 0) {
            sx_m[8 * warp + r4] = m_w;
            sx_l[8 * warp + r4] = lq;
            if (warp == 0) sx_ref[r4] = ref;
        }
    }
    __syncthreads();
    float M = -INFINITY;  // -inf only for an item without tokens
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sx_m[8 * w + r4]);
    float lsum = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) lsum += sx_l[8 * w + r4] * exp2_diff(sx_m[8 * w + r4], M);
    const uint32_t refb = sx_ref[r4];
    {
        // v~ = sum over the group's warps of 2^(m_w - M) v~_w, gathered in its
        // warp 0.  The other warps' scaled values pass through a slot that is
        // free by now: a chunk's P^V fits one piece (ranks <= d), so after its
        // last C piece no copy targets that slot (each group has its own part
        // of it); a tail group's values pass through its own slot, whose data
        // it has consumed.
        constexpr int kXV = (kWarps - 1) * (D / 8) * 32 * 16;  // one group's exchange
        static_assert(RG * kXV <= kPieceBytes, "warp values fit a slot");
        static_assert(L::kRanksPerPiece >= D, "P^V of any rank is one piece");
        const float sc = exp2_diff(m_w, M);
        // (reading an INT8 plan: the bf16 slot, whose next read-back, of
        // P^V, comes after the exchange)
        const int free_slot = Q8 ? 1 : (ps.npk + ps.nc - 1) & 1;
        float4 *xv = reinterpret_cast<float4 *>(smem + (is_tail ? grp * kPieceBytes
                                                                : free_slot * kPieceBytes + grp * kXV));
        if (warp > 0) {
#pragma unroll
            for (int n = 0; n < NT; ++n)
                xv[((warp - 1) * NT + n) * 32 + lane] =
                    make_float4(sc * vacc[n][0], sc * vacc[n][1], sc * vacc[n][2], sc * vacc[n][3]);
        }
        __syncthreads();
        if (warp == 0) {
#pragma unroll
            for (int n = 0; n < NT; ++n) {
                float4 a = make_float4(sc * vacc[n][0], sc * vacc[n][1], sc * vacc[n][2], sc * vacc[n][3]);
#pragma unroll
                for (int w = 1; w < kWarps; ++w) {
                    const float4 o = xv[((w - 1) * NT + n) * 32 + lane];
                    a.x += o.x;
                    a.y += o.y;
                    a.z += o.z;
                    a.w += o.w;
                }
                vacc[n][0] = a.x;
                vacc[n][1] = a.y;
                vacc[n][2] = a.z;
                vacc[n][3] = a.w;
            }
        }
    }

    bool direct;
    int64_t rec_idx;
    int row0, nrows;
    if (is_tail) {
        // the values are already in the head dimension: o = v~ (warp 0 adds all of it)
        rec_idx = p.tail_rec_base + item;
        row0 = qi * p.G + 8 * rq;
        nrows = active ? min(8, p.G - 8 * rq) : 0;
        float ov[NT][2];
#pragma unroll
        for (int n = 0; n < NT; ++n) {
            ov[n][0] = vacc[n][0] + vacc[n][2];
            ov[n][1] = vacc[n][1] + vacc[n][3];
        }
        direct = warp == 0 ? add_part<D, NT>(p, g, lane, 0, ov, M, lsum, refb, true, row0, nrows, rec_idx)
                           : __all_sync(0xffffffffu, r4 >= nrows || !(M - (refb ? ref_dec(refb) : M) > kDirectMax));
    } else {
        rec_idx = RG == 1 ? (int64_t)blockIdx.x : (int64_t)(blockIdx.x / nrgb) * p.nrg + rgrp;
        row0 = 8 * rgrp;
        nrows = active ? min(8, p.rows_g - row0) : 0;
        // warp 0 stages the merged v~ as the back-projection's A fragments (rows
        // 0-7 hi, 8-15 lo) in the q~ area, so that the rank loop below stays rolled
        if (warp == 0) {
#pragma unroll
            for (int ks = 0; ks < NT / 2; ++ks) {
                uint4 f;
                split_hi_lo(vacc[2 * ks][0] + vacc[2 * ks][2], vacc[2 * ks][1] + vacc[2 * ks][3], f.x, f.y);
                split_hi_lo(vacc[2 * ks + 1][0] + vacc[2 * ks + 1][2], vacc[2 * ks + 1][1] + vacc[2 * ks + 1][3],
                            f.z, f.w);
                sq[ks * 32 + lane] = f;
            }
        }
        __syncthreads();
        // back-projection: warp w produces head-dimension columns [w D / kWarps, (w + 1) D / kWarps)
        constexpr int NO = NT / kWarps;  // 8-column tiles per warp
        static_assert(NO % 2 == 0, "column pairs per warp");
        float o[NO][4];
#pragma unroll
        for (int n = 0; n < NO; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
#pragma unroll 1
        for (int k = ps.npk + ps.nc; k < np; ++k) {
            const uint32_t slot = wait_piece(k);
            // rank 8-groups [r0, r1) of this piece: 16-rank k-steps of v~
            const int r0 = (k - ps.npk - ps.nc) * ps.rpp, r1 = min(r0 + ps.rpp, nrv);
#pragma unroll 1
            for (int ks = r0 / 2; active && 2 * ks < r1; ++ks) {
                const uint4 a4 = sq[ks * 32 + lane];
                const uint32_t a[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                for (int cp = 0; cp < NO / 2; ++cp) {
                    // matrices (transposed): (2ks, 2c), (2ks + 1, 2c), (2ks, 2c + 1), (2ks + 1, 2c + 1)
                    const int jg = 2 * ks + (mi & 1), cg = warp * NO + 2 * cp + (mi >> 1);
                    const uint32_t addr = jg < r1 ? slot + ((jg - r0) * NT + cg) * 128 + mr * 16 : zline;
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_t(addr, b0, b1, b2, b3);
                    mma16816(o[2 * cp], a, b0, b1);
                    mma16816(o[2 * cp + 1], a, b2, b3);
                }
            }
            release_piece(k);
        }
        float ov[NO][2];
#pragma unroll
        for (int n = 0; n < NO; ++n) {
            ov[n][0] = o[n][0] + o[n][2];
            ov[n][1] = o[n][1] + o[n][3];
        }
        direct = add_part<D, NO>(p, g, lane, warp * NO, ov, M, lsum, refb, warp == 0, row0, nrows, rec_idx);
    }

    // ---- an outlier's record is listed; the finish grid that follows
    // (programmatic dependent launch) sees every reduction and record
    if (leader && active && !direct) {
        // in the list of every row group the item's rows touch
        for (int rg = row0 / 8; rg <= (row0 + nrows - 1) / 8; ++rg) {
            const int gr = g * p.nrg + rg;
            const uint32_t k = atomicAdd(p.ovf_cnt + gr, 1u);
            __stcg(reinterpret_cast<int4 *>(p.ovf_list) + (int64_t)gr * p.list_cap + k,
                   make_int4((int)rec_idx, row0, nrows, 0));
        }
    }
}

// One warp per (KV head, group of 8 query rows): normalise the accumulators
// once the chunk grid is done.
template <int D>
__global__ void __launch_bounds__(32) finish_kernel(const __grid_constant__ DecodeParams p)
{
    pdl_trigger();
    pdl_wait();  // the chunk grid's reductions and records are visible from here
    finish_head<D>(p, blockIdx.x / p.nrg, blockIdx.x % p.nrg, threadIdx.x);
}

}  // namespace

namespace {
template <int D, int RG, bool Q8>
cudaError_t launch_chunk_grid(cudaLaunchConfig_t cfg, const DecodeParams &p, const CUtensorMap &mk,
                              const CUtensorMap &mv)
{
    using L = CLay<D, RG>;
    constexpr int kSmem = Q8 ? L::kTotalQ8 : L::kTotal;
    static bool configured[kMaxDevices] = {};
    const int dev = attribute_slot();
    if (dev < 0 || !configured[dev]) {
        cudaError_t e = cudaFuncSetAttribute(chunk_kernel<D, RG, Q8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSmem);
        if (e != cudaSuccess) return e;
        // several thread blocks per SM need the largest shared-memory carveout
        e = cudaFuncSetAttribute(chunk_kernel<D, RG, Q8>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        if (e != cudaSuccess) return e;
        if (dev >= 0) configured[dev] = true;
    }
    const int nrgb = (p.nrg + RG - 1) / RG;
    cfg.gridDim = dim3(p.num_chunks * nrgb + (p.has_tail ? (p.num_tail_items + RG - 1) / RG : 0));
    cfg.blockDim = dim3(32 * kWarpsOf<RG> * RG);
    cfg.dynamicSmemBytes = (size_t)kSmem;
    return cudaLaunchKernelEx(&cfg, chunk_kernel<D, RG, Q8>, p, mk, mv);
}

template <int D, bool Q8>
cudaError_t launch_chunk_grid_d(cudaLaunchConfig_t cfg, const DecodeParams &p, const CUtensorMap &mk,
                                const CUtensorMap &mv)
{
    // two row groups per block once a KV head has more than 8 query rows
    // (one when the grid holds long tail items alone)
    const bool two = p.nrg >= 2 && p.tail_pieces <= 1;
    return two ? launch_chunk_grid<D, 2, Q8>(cfg, p, mk, mv) : launch_chunk_grid<D, 1, Q8>(cfg, p, mk, mv);
}
}  // namespace

cudaError_t launch_chunks(const DecodeParams &p, const void *tmap_k, const void *tmap_v, cudaStream_t stream)
{
    const CUtensorMap &mk = *static_cast<const CUtensorMap *>(tmap_k);
    const CUtensorMap &mv = *static_cast<const CUtensorMap *>(tmap_v);
    cudaLaunchConfig_t cfg = {};
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // (an INT8 plan read directly: the INT8 variant; its tail items are bf16)
    const bool q8 = p.q8_codes != nullptr;
    cudaError_t e = p.d == 64 ? (q8 ? launch_chunk_grid_d<64, true>(cfg, p, mk, mv)
                                    : launch_chunk_grid_d<64, false>(cfg, p, mk, mv))
                              : (q8 ? launch_chunk_grid_d<128, true>(cfg, p, mk, mv)
                                    : launch_chunk_grid_d<128, false>(cfg, p, mk, mv));
    if (e != cudaSuccess) return e;
    // the tensor-core and reconstruct-then-attend calls launch their prefix
    // grid between the two
    if (p.tc_ntile > 0 || p.rc_chunks) return cudaSuccess;
    return launch_finish(p, stream);
}

cudaError_t launch_finish(const DecodeParams &p, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(p.hkv * p.nrg);
    cfg.blockDim = dim3(32);
    cfg.dynamicSmemBytes = 0;
    return p.d == 64 ? cudaLaunchKernelEx(&cfg, finish_kernel<64>, p) : cudaLaunchKernelEx(&cfg, finish_kernel<128>, p);
}

}  // namespace milo
