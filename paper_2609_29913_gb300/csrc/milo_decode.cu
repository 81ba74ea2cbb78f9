// milo_decode.cu -- decode attention over a block-wise low-rank KV prefix
// (MILO, Alg. 1 Stage 2 + Eq. 1), computed in each block's rank space:
//
//   scores  s_t = scale * <q, K^_b[t]> = <C^K_b[t,:], scale * P^K_b q>   (Eq. 3 into Eq. 1)
//   values  sum_t p_t V^_b[t] = (sum_t p_t C^V_b[t,:]) P^V_b
//
// followed by the query's dense tail and an exact log-sum-exp merge of the
// split softmax (Eq. 1 is associative over token partitions once each part
// carries its running max and sum).
//
// This file holds the persistent kernel, used when more than 8 query heads
// share a KV head (G > 8; several row groups share every coefficient tile
// read) or a plan has no prefix, and the merge kernel.  Every other call
// takes the chunk grid of milo_chunk.cu.
//
// Persistent kernel, one thread block per SM, two roles:
//   producer   (warp 0, one lane): turns the block's static list of prefix
//              segments, then dynamically claimed dense-tail items, into an
//              in-order stream of "fills" of at most kSlotBytes.  A fill packs
//              the previous segment's P^V, the next segment's P^K and as many
//              whole coefficient tiles of that segment as fit; a tail fill
//              holds one tail item's K and V (3-D TMA).  Each fill is one ring
//              slot, one mbarrier, up to six bulk copies.
//   MMA warps  (warps 1..7): consume every fill in order.  P^K part: each warp
//              projects q~ = scale * log2(e) * P^K q for a slice of the rank
//              tiles (mma m16n8k16, result split into bf16 hi + lo rows).
//              Coefficient part: 32-token tiles round-robin over the warps --
//              scores (A rows 0-7 q~ hi, rows 8-15 q~ lo), online softmax in
//              registers, rank-space values (A rows = p hi, p lo).  P^V part
//              (segment end): the warps pool their (max, sum, v~), each merges
//              a slice of v~, then each back-projects a slice of the head
//              dimension through P^V into its running output; at the end of a
//              run the slices are written as one partial record.  Tail fills
//              go whole to one warp each.
// The merge kernel (launched next, with programmatic dependent launch)
// combines the partial records of every (KV head, row group).  Every wait is
// bounded (~2 s); on expiry the thread records MILO_ERR_TIMEOUT in the sticky
// status word and leaves.
#include <cuda.h>
#include <cuda_bf16.h>

#include <mutex>
#include <type_traits>

#include "milo.h"
#include "milo_internal.h"
#include "milo_ptx.cuh"

namespace milo {
namespace {

// run flags of a segment end
enum : int { F_RUN_FIRST = 1, F_RUN_LAST = 2 };
// barrier indices: full[kSlots], empty[kSlots], then the MMA warps' own
enum : int {
    B_GS = 2 * kSlots,  // group sync of the MMA warps
    B_QREADY,           // [2] q~ buffer written by every MMA warp
    B_QFREE = B_QREADY + 2,  // [2] q~ buffer loaded by every MMA warp
    B_DUMPED = B_QFREE + 2,  // every MMA warp dumped its state of a segment
    B_MERGED,           // every MMA warp merged its slice of the pooled v~
    B_BPDONE,           // every MMA warp back-projected (merged v~ buffer free)
    B_COUNT
};

// ------------------------------------------------------- shared memory ----
constexpr int al(int x, int a) { return (x + a - 1) / a * a; }
template <int D>
struct Lay {
    static constexpr int kRing = 0;                               // kSlots fills
    static constexpr int kMerge = kRing + kSlots * kSlotBytes;    // per-warp (max, sum, v~) dumps
    static constexpr int kMergeWarp = 32 * D + 256;               // v~ [d/8][32 lanes] float2 + (m,l) [32] float2
    static constexpr int kFragPart = (D / 16) * 32 * 16;          // A fragments (hi/lo) of one row group
    static constexpr int kQs = kMerge + kMmaWarps * kMergeWarp;   // q~ [2 buffers][2 row groups]
    static constexpr int kAf = kQs + 4 * kFragPart;               // merged v~ of two row groups
    static constexpr int kHdr = kAf + 2 * kFragPart;
    static constexpr int kQc = al(kHdr + kSlots * kHdrInts * 4, 128);  // copy of q when it is small
    static constexpr int kQcBytes = 8192;
    static constexpr int kBar = kQc + kQcBytes;
    static constexpr int kZero = al(kBar + B_COUNT * 8, 128);
    static constexpr int kTotal = kZero + 128;
    static_assert(kSlotBytes % 1024 == 0, "ring slots must keep 1024-byte alignment (128B-swizzled TMA boxes)");
    static_assert(kMerge % 128 == 0 && kQs % 128 == 0 && kAf % 128 == 0 && kHdr % 128 == 0, "alignment");
    static_assert(kQc % 128 == 0 && kBar % 128 == 0, "alignment");
    static_assert(2 * D * kTailTokens * 2 <= kSlotBytes, "a tail item must fit one fill");
    static_assert(D * D * 2 <= kSlotBytes, "a full-rank basis must fit one fill");
    static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// Iterator over a thread block's prefix work in emission order:
// run (consecutive segments of one KV head) -> row-group pass -> segment.
struct SegIter {
    int r0, r1, pass, sg, s_end;
    bool done;
    __device__ void find_run_end(const DecodeParams &p)
    {
        r1 = r0;
        while (r1 < s_end - 1 && !(p.segs[r1].flags & kSegLastOfRun)) ++r1;
    }
    __device__ void begin(const DecodeParams &p, int s_begin, int s_end_)
    {
        s_end = s_end_;
        r0 = s_begin;
        pass = 0;
        sg = s_begin;
        done = s_begin >= s_end;
        if (!done) find_run_end(p);
    }
    __device__ void advance(const DecodeParams &p)
    {
        if (sg < r1) {
            ++sg;
        } else if (pass + 1 < p.npass) {
            ++pass;
            sg = r0;
        } else {
            r0 = r1 + 1;
            pass = 0;
            sg = r0;
            done = r0 >= s_end;
            if (!done) find_run_end(p);
        }
    }
};

// ================================================================ producer
template <int D>
__device__ void run_producer(const DecodeParams &p, uint8_t *smem, int32_t *hdr, uint64_t *bars,
                             const CUtensorMap *tmap_k, const CUtensorMap *tmap_v)
{
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    // a tail item lands as cores [column group][token group] (one 16-byte column
    // chunk per box), the layout of a packed coefficient tile
    constexpr uint32_t kTailChunk = kTailTokens * 16;             // one box: kTailTokens rows x 8 columns
    constexpr uint32_t kTailBytes = 2 * (D / 8) * kTailChunk;
    int seq = 0;
    bool ok = true;

    // the fill under construction
    int slot = 0, flags = 0, ncp = 0;
    uint32_t used = 0;
    int32_t *h = nullptr;
    uint32_t cp_off[6], cp_bytes[6];
    const uint8_t *cp_src[6];
    int tail_row = -1, tail_g = 0;

    auto open_fill = [&]() -> bool {
        slot = seq % kSlots;
        if (seq >= kSlots && !mbar_wait(bar(kSlots + slot), ((seq / kSlots) - 1) & 1, p.status)) return false;
        h = hdr + slot * kHdrInts;
        used = 0;
        flags = 0;
        ncp = 0;
        tail_row = -1;
        return true;
    };
    auto add_copy = [&](uint32_t off, const uint8_t *src, uint32_t bytes) {
        if (bytes == 0) return;
        cp_off[ncp] = off;
        cp_src[ncp] = src;
        cp_bytes[ncp] = bytes;
        ++ncp;
    };
    auto close_fill = [&]() {
        h[H_FLAGS] = flags;
        const uint32_t fb = bar(slot);
        uint32_t tx = tail_row >= 0 ? kTailBytes : 0u;
        for (int c = 0; c < ncp; ++c) tx += cp_bytes[c];
        const uint32_t base = smem_u32(smem + Lay<D>::kRing + slot * kSlotBytes);
        if (tx) {
            mbar_arrive_tx(fb, tx);
            for (int c = 0; c < ncp; ++c) bulk_g2s(base + cp_off[c], cp_src[c], cp_bytes[c], fb);
            if (tail_row >= 0) {
#pragma unroll 1
                for (int c = 0; c < D / 8; ++c) {
                    tma_load_3d(base + c * kTailChunk, tmap_k, 8 * c, tail_g, tail_row, fb);
                    tma_load_3d(base + (D / 8 + c) * kTailChunk, tmap_v, 8 * c, tail_g, tail_row, fb);
                }
            }
        } else {
            mbar_arrive(fb);
        }
        ++seq;
    };

    // P^V of the last finished segment, attached to the next fill
    bool pv_pending = false;
    int pv_g = 0, pv_rv8 = 0, pv_rec = 0, pv_run = 0, pv_pass = 0, pv_seg = 0;
    int64_t pv_off = 0;
    auto put_pv = [&]() {
        const uint32_t bytes = (uint32_t)pv_rv8 * D * 2;
        h[H_PV_G] = pv_g;
        h[H_PV_RV8] = pv_rv8;
        h[H_PV_REC] = pv_rec;
        h[H_PV_SEG] = pv_seg;
        h[H_PV_RUN] = pv_run;
        h[H_PV_PASS] = pv_pass;
        h[H_PV_OFF] = (int)used;
        add_copy(used, p.packed + pv_off, bytes);
        used += bytes;
        flags |= kHasPv;
        pv_pending = false;
    };
    auto flush_pv = [&]() -> bool {
        if (!pv_pending) return true;
        if (!open_fill()) return false;
        put_pv();
        close_fill();
        return true;
    };

    // P^K goes out one segment early (the MMA warps project while the previous
    // segment streams); pk_it walks the (segment, pass) sequence ahead of it
    SegIter pk_it;
    int pk_j = 0;
    auto put_pks = [&](int j) {
        for (int part = 0; part < 2 && !pk_it.done && pk_j <= j + 1; ++part) {
            const EntryDev e = p.entries[p.segs[pk_it.sg].entry];
            const int rk8 = (e.rk + 7) & ~7;
            const uint32_t bytes = (uint32_t)rk8 * D * 2;
            if (used + bytes > (uint32_t)kSlotBytes) return;
            int32_t *f = h + H_PK_J + 5 * part;
            f[0] = pk_j;
            f[1] = e.g;
            f[2] = rk8;
            f[3] = pk_it.pass;
            f[4] = (int)used;
            add_copy(used, p.packed + e.off_pk, bytes);
            used += bytes;
            flags |= part == 0 ? kHasPk0 : kHasPk1;
            ++pk_j;
            pk_it.advance(p);
        }
    };

    auto emit_segment = [&](const SegIter &it, int j) -> bool {
        const SegDev seg = p.segs[it.sg];
        const EntryDev ent = p.entries[seg.entry];
        const int rk8 = (ent.rk + 7) & ~7, rv8 = (ent.rv + 7) & ~7;
        const int n8 = (ent.n + 7) & ~7;
        bool started = false;
        int t = seg.t0;
        while (!started || t < seg.t1) {
            if (!open_fill()) return false;
            if (pv_pending) put_pv();
            put_pks(j);
            if (!started) {
                if (pk_j <= j) {  // this segment's basis has not gone out yet
                    close_fill();
                    continue;
                }
                h[H_SS_J] = j;
                h[H_SS_PASS] = it.pass;
                h[H_SS_RK8] = rk8;
                flags |= kSegStart;
                started = true;
            }
            if (t < seg.t1) {
                // whole coefficient tiles (the entry's last one may be short)
                const uint32_t cap = (uint32_t)kSlotBytes - used;
                int tt1 = t;
                uint32_t cbytes = 0;
                while (tt1 < seg.t1) {
                    const int te = min(tt1 + kTileTokens, seg.t1);
                    const int tok = min((te + 7) & ~7, n8) - tt1;
                    const uint32_t b = (uint32_t)tok * (rk8 + rv8) * 2;
                    if (cbytes + b > cap) break;
                    cbytes += b;
                    tt1 = te;
                }
                if (tt1 > t) {
                    const int tok8 = min((tt1 + 7) & ~7, n8) - t;
                    const uint32_t kb = (uint32_t)tok8 * rk8 * 2, vb = (uint32_t)tok8 * rv8 * 2;
                    h[H_C_OFF] = (int)used;
                    h[H_T0] = t;
                    h[H_T1] = tt1;
                    h[H_RK8] = rk8;
                    h[H_RV8] = rv8;
                    h[H_TOK8] = tok8;
                    add_copy(used, p.packed + ent.off_ck + (int64_t)t * rk8 * 2, kb);
                    add_copy(used + kb, p.packed + ent.off_cv + (int64_t)t * rv8 * 2, vb);
                    used += kb + vb;
                    flags |= kHasC;
                    t = tt1;
                }
            }
            close_fill();
        }
        pv_pending = true;
        pv_g = ent.g;
        pv_rv8 = rv8;
        pv_rec = seg.slot;
        pv_seg = it.sg;
        pv_run = (it.sg == it.r0 ? F_RUN_FIRST : 0) | (it.sg == it.r1 ? F_RUN_LAST : 0);
        pv_pass = it.pass;
        pv_off = ent.off_pv;
        return true;
    };

    auto emit_tail = [&](uint32_t item) -> bool {
        if (!flush_pv()) return false;
        const int S = p.tail_splits;
        const int i = item / (p.hkv * S), g = (item / S) % p.hkv, sp = item % S;
        const int64_t o0 = p.tail_offsets[i], o1 = p.tail_offsets[i + 1];
        const int T = (int)(o1 - o0);
        if (sp == S - 1 && T > S * kTailTokens) atomicCAS(p.status, 0, (int32_t)MILO_ERR_DEVICE_BOUNDS);
        const int t0 = sp * kTailTokens, t1 = min(t0 + kTailTokens, T);
        if (!open_fill()) return false;
        h[H_QI] = i;
        h[H_G] = g;
        h[H_ITEM] = (int)item;
        h[H_T0] = t0;
        h[H_T1] = t1;
        flags |= kTailFill;
        if (t1 > t0) {
            tail_row = (int)(o0 + t0);
            tail_g = g;
        }
        close_fill();
        return true;
    };
    auto grab_tails = [&](uint32_t max_items) -> bool {
        if (!p.has_tail) return true;
        for (uint32_t n = 0; n < max_items; ++n) {
            const uint32_t item = atomicAdd(&p.counters->tail_next, 1u);
            if (item >= (uint32_t)p.num_tail_items) return true;
            if (!emit_tail(item)) return false;
        }
        return true;
    };

    const int cta = blockIdx.x;
    SegIter it;
    it.begin(p, p.cta_seg_begin[cta], p.cta_seg_begin[cta + 1]);
    pk_it = it;
    for (int j = 0; ok && !it.done; ++j) {
        ok = emit_segment(it, j);
        it.advance(p);
    }
    // tail items go after the prefix (any block that finishes early takes more);
    // the tail counter and the tails belong to the preceding grid until here
    pdl_wait();
    if (ok) ok = grab_tails(0xffffffffu);
    if (ok && open_fill()) {
        if (pv_pending) put_pv();
        flags |= kEndFill;
        close_fill();
    }
    // the last thread block to finish grabbing resets the tail counter
    if (atomicAdd(&p.counters->ctas_done, 1u) == (uint32_t)p.num_ctas - 1) {
        p.counters->tail_next = 0u;
        p.counters->ctas_done = 0u;
    }
    // do not leave while a copy this thread started may still be landing
    for (int j = max(0, seq - kSlots); j < seq; ++j)
        if (!mbar_wait(bar(j % kSlots), (j / kSlots) & 1, p.status)) break;
}

// ================================================================ MMA warps
template <int N>
using IC = std::integral_constant<int, N>;

template <int D>
__device__ bool run_mma(const DecodeParams &p, uint8_t *smem, const int32_t *hdr, uint64_t *bars, uint32_t zero_addr,
                        int mw, int lane)
{
    using L = Lay<D>;
    constexpr int kMaxNt = D / 8;   // max rank (or column) 8-tiles
    constexpr int kMaxKs = D / 16;  // max 16-wide k-steps
    // column tiles one warp back-projects (a row group has at least kMmaWarps / 2
    // warps), rounded up to even: the back-projection takes them in pairs
    constexpr int kMaxCt = ((kMaxNt + kMmaWarps / 2 - 1) / (kMmaWarps / 2) + 1) & ~1;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    const int quad = lane / 4, qlane = lane % 4, mi = lane / 8;
    const int recf = 8 * D + kRecFloatsExtra;
    // prefix row groups: warp mw serves group mw % ngrp as member wi of nwg
    const int ngrp = p.nrg_cta, grp = mw % ngrp, wi = mw / ngrp;
    const int nwg = (kMmaWarps - grp + ngrp - 1) / ngrp;
    float2 *myregion = reinterpret_cast<float2 *>(smem + L::kMerge + mw * L::kMergeWarp);
    auto region = [&](int w) { return reinterpret_cast<const float2 *>(smem + L::kMerge + w * L::kMergeWarp); };
    auto qs_part = [&](int b) { return reinterpret_cast<uint32_t *>(smem + L::kQs + (2 * b + grp) * L::kFragPart); };
    uint32_t *af = reinterpret_cast<uint32_t *>(smem + L::kAf + grp * L::kFragPart);
    const bool qcached = (int64_t)p.batch * p.hq * D * 2 <= L::kQcBytes;
    const uint16_t *qsrc = qcached ? reinterpret_cast<const uint16_t *>(smem + L::kQc) : p.q;

    // A operand of the scores, read per tile: hi/lo fragments of q~ (a q~ buffer)
    // or of scale * log2(e) * q for a tail item (this warp's dump area)
    uint32_t a_frag = 0;
    int cur_b = 0;      // q~ buffer of the current segment
    float vacc[kMaxNt][4];
    float m_w = -INFINITY, l_w = 0.f;
    float orun[kMaxCt][2];
    float m_run = -INFINITY, l_run = 0.f;
    bool act = false;   // this warp's row group exists in the current pass
    int ngs = 0;        // group syncs passed
    int tile_base = 0;  // round-robin position of prefix tiles
    int tail_ctr = 0;   // tail row-group jobs seen
    int nends = 0;      // segment ends so far (the same count in every MMA warp)
    // the pending segment end: 0 none, 1 merge next, 2 back-projection next
    int pend = 0, pe_e = 0, pe_seq = 0, pe_g = 0, pe_rg = 0, pe_rv8 = 0, pe_run = 0, pe_rec = 0;
    uint32_t pe_pv = 0;
    float pe_M = -INFINITY, pe_arun = 0.f, pe_Ls = 0.f;
#pragma unroll
    for (int c = 0; c < kMaxCt; ++c) orun[c][0] = orun[c][1] = 0.f;

    auto gsync = [&]() -> bool {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(B_GS));
        const bool ok = warp_wait(bar(B_GS), ngs & 1, p.status);
        ++ngs;
        return ok;
    };
    auto arrive = [&](int b) {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(b));
    };
    auto test_bar = [&](int b, int parity) -> bool {
        int ok = 0;
        if (lane == 0) ok = mbar_test(bar(b), parity) ? 1 : 0;
        return __shfl_sync(0xffffffffu, ok, 0) != 0;
    };
    auto reset_state = [&]() {
        m_w = -INFINITY;
        l_w = 0.f;
#pragma unroll
        for (int x = 0; x < kMaxNt; ++x) vacc[x][0] = vacc[x][1] = vacc[x][2] = vacc[x][3] = 0.f;
    };
    // The tile code comes in four widths (1, 2, 4 and D/16 k-steps of 16 ranks;
    // rank groups past a factor's rank read a zero line): close to the exact
    // work for every rank, while the hot code stays small enough for the
    // instruction cache (which a variant per rank overflows).
    auto full_width = [&](int /*nk*/, auto body) { body(IC<kMaxKs>{}); };
    auto by_width = [&](int nk, auto body) {
        if (nk <= 1) body(IC<1>{});
        else if (nk <= 2) body(IC<2>{});
        else if (nk <= 4) body(IC<4>{});
        else body(IC<kMaxKs>{});
    };

    // One 32-token tile (token groups 0-3) with NK 16-wide k-steps: scores,
    // online softmax, rank-space values.  Keys/values are read through
    // kaddr(h, m, kk) / vaddr(h, m, jp), h = half of the tile (token groups 2h, 2h+1).
    auto tile32 = [&](auto nkc, float sc_mul, int tok_base, int t1, int ntg, auto kaddr, auto vaddr) {
        constexpr int NK = decltype(nkc)::value;
        float sc4[4][4];
#pragma unroll
        for (int n = 0; n < 4; ++n) sc4[n][0] = sc4[n][1] = sc4[n][2] = sc4[n][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < NK; ++kk) {
            uint32_t qa[4];
            asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                         : "=r"(qa[0]), "=r"(qa[1]), "=r"(qa[2]), "=r"(qa[3])
                         : "r"(a_frag + (kk * 32 + lane) * 16));
            uint32_t b0, b1, b2, b3, c0, c1, c2, c3;
            ldsm_x4(kaddr(0, mi, kk), b0, b1, b2, b3);
            ldsm_x4(kaddr(1, mi, kk), c0, c1, c2, c3);
            mma16816(sc4[0], qa, b0, b1);
            mma16816(sc4[1], qa, b2, b3);
            mma16816(sc4[2], qa, c0, c1);
            mma16816(sc4[3], qa, c2, c3);
        }
        // score of token tok_base + 8n + 2 qlane + j (rows: hi part + lo part)
        float sv[8];
#pragma unroll
        for (int n = 0; n < 4; ++n) {
            const int tok = tok_base + 8 * n + 2 * qlane;
            sv[2 * n] = (n < ntg && tok < t1) ? (sc4[n][0] + sc4[n][2]) * sc_mul : -INFINITY;
            sv[2 * n + 1] = (n < ntg && tok + 1 < t1) ? (sc4[n][1] + sc4[n][3]) * sc_mul : -INFINITY;
        }
        float mx = sv[0];
#pragma unroll
        for (int j = 1; j < 8; ++j) mx = fmaxf(mx, sv[j]);
        mx = quad_max(mx);
        if (mx > m_w + 8.f) {  // lazy rescale: p stays <= 2^8
            const float alpha = exp2_diff(m_w, mx);
            l_w *= alpha;
#pragma unroll
            for (int x = 0; x < 2 * NK; ++x) {
                vacc[x][0] *= alpha; vacc[x][1] *= alpha; vacc[x][2] *= alpha; vacc[x][3] *= alpha;
            }
            m_w = mx;
        }
        float pv[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) pv[j] = exp2f(sv[j] - m_w);
        l_w += ((pv[0] + pv[1]) + (pv[2] + pv[3])) + ((pv[4] + pv[5]) + (pv[6] + pv[7]));
        uint32_t pa0[4], pa1[4];
        split_hi_lo(pv[0], pv[1], pa0[0], pa0[1]);
        split_hi_lo(pv[2], pv[3], pa0[2], pa0[3]);
        split_hi_lo(pv[4], pv[5], pa1[0], pa1[1]);
        split_hi_lo(pv[6], pv[7], pa1[2], pa1[3]);
#pragma unroll
        for (int jp = 0; jp < NK; ++jp) {
            uint32_t b0, b1, b2, b3, c0, c1, c2, c3;
            ldsm_x4_t(vaddr(0, mi, jp), b0, b1, b2, b3);
            ldsm_x4_t(vaddr(1, mi, jp), c0, c1, c2, c3);
            mma16816(vacc[2 * jp], pa0, b0, b1);
            mma16816(vacc[2 * jp + 1], pa0, b2, b3);
            mma16816(vacc[2 * jp], pa1, c0, c1);
            mma16816(vacc[2 * jp + 1], pa1, c2, c3);
        }
    };

    // ---- segment end, deferred in three steps: dump (at the P^V part), merge
    // slice (once every warp dumped), back-projection (once every warp merged).
    // The fill carrying P^V stays held until this warp's back-projection.
    auto do_merge = [&]() -> bool {
        // the merged v~ buffer is free once every warp back-projected the previous end
        if (pe_e >= 1 && !warp_wait(bar(B_BPDONE), (pe_e - 1) & 1, p.status)) return false;
        const bool pact = pe_rg < p.nrg;
        const int nvt = pe_rv8 / 8, nkj = (pe_rv8 + 15) / 16;
        if (pe_run & F_RUN_FIRST) {
            m_run = -INFINITY;
            l_run = 0.f;
#pragma unroll
            for (int c = 0; c < kMaxCt; ++c) orun[c][0] = orun[c][1] = 0.f;
        }
        // merge weights relative to the run's new maximum (row = quad); another row
        // group's dumps may hold anything: select, never multiply by zero
        float2 ml[kMmaWarps];
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w) ml[w] = region(w)[kMaxNt * 32 + lane];
        float M = m_run;
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w)
            if ((w & (ngrp - 1)) == grp) M = fmaxf(M, ml[w].x);
        float sc[kMmaWarps];
        float Ls = 0.f;
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w) {
            const bool mine = (w & (ngrp - 1)) == grp;
            sc[w] = mine ? exp2_diff(ml[w].x, M) : 0.f;
            Ls += mine ? sc[w] * ml[w].y : 0.f;
        }
        // this warp's slice of the merged v~ (tiles wi, wi + nwg, ...), as bf16 hi/lo A fragments
#pragma unroll 1
        for (int x = wi; x < 2 * nkj; x += nwg) {
            {
                float2 t[kMmaWarps];
#pragma unroll
                for (int w = 0; w < kMmaWarps; ++w) t[w] = region(w)[x * 32 + lane];
                float2 v = make_float2(0.f, 0.f);
#pragma unroll
                for (int w = 0; w < kMmaWarps; ++w) {
                    const bool mine = (w & (ngrp - 1)) == grp;
                    v.x = mine ? fmaf(sc[w], t[w].x, v.x) : v.x;
                    v.y = mine ? fmaf(sc[w], t[w].y, v.y) : v.y;
                }
                if (!(pact && x < nvt)) v = make_float2(0.f, 0.f);
                uint32_t hi, lo;
                split_hi_lo(v.x, v.y, hi, lo);
                af[((x / 2) * 32 + lane) * 4 + (x & 1) * 2 + 0] = hi;
                af[((x / 2) * 32 + lane) * 4 + (x & 1) * 2 + 1] = lo;
            }
        }
        pe_M = M;
        pe_arun = exp2_diff(m_run, M);
        pe_Ls = Ls;
        arrive(B_MERGED);
        pend = 2;
        return true;
    };
    auto do_backproj = [&]() {
        const bool pact = pe_rg < p.nrg;
        const int nvt = pe_rv8 / 8;
        if (pact) {
            full_width((pe_rv8 + 15) / 16, [&](auto nkc) {
                float o[kMaxCt][4];
#pragma unroll
                for (int c = 0; c < kMaxCt; ++c) o[c][0] = o[c][1] = o[c][2] = o[c][3] = 0.f;
#pragma unroll 1
                for (int kj = 0; kj < (pe_rv8 + 15) / 16; ++kj) {
                    const uint4 a4 = reinterpret_cast<const uint4 *>(af)[kj * 32 + lane];
                    const uint32_t a[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                    for (int cp = 0; cp < kMaxCt; cp += 2) {
                        if (wi + cp * nwg < kMaxNt) {
                            const int ct = wi + (cp + (mi >> 1)) * nwg;  // matrices 2,3: the pair's second tile
                            const int jg = 2 * kj + (mi & 1);
                            const uint32_t addr = (ct < kMaxNt && jg < nvt)
                                                      ? pe_pv + (jg * (D / 8) + ct) * 128 + (lane % 8) * 16
                                                      : zero_addr;
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4_t(addr, b0, b1, b2, b3);
                            mma16816(o[cp], a, b0, b1);
                            mma16816(o[cp + 1], a, b2, b3);
                        }
                    }
                }
#pragma unroll
                for (int c = 0; c < kMaxCt; ++c) {
                    orun[c][0] = orun[c][0] * pe_arun + (o[c][0] + o[c][2]);
                    orun[c][1] = orun[c][1] * pe_arun + (o[c][1] + o[c][3]);
                }
            });
            l_run = l_run * pe_arun + pe_Ls;
            m_run = pe_M;
            if (pe_run & F_RUN_LAST) {
                float *rec = p.rec + ((int64_t)pe_rec * p.nrg + pe_rg) * recf;
#pragma unroll
                for (int c = 0; c < kMaxCt; ++c)
                    if (wi + c * nwg < kMaxNt)
                        __stcg(reinterpret_cast<float2 *>(rec + quad * D + 8 * (wi + c * nwg) + 2 * qlane),
                               make_float2(orun[c][0], orun[c][1]));
                if (wi == 0 && qlane == 0) {
                    __stcg(rec + 8 * D + quad, m_run);
                    __stcg(rec + 8 * D + 8 + quad, l_run);
                }
            }
        }
        arrive(kSlots + pe_seq % kSlots);  // the fill that carried P^V
        arrive(B_BPDONE);
        pend = 0;
    };
    // Advance the pending segment end as far as the other warps allow
    // (force: wait for them).
    auto poll = [&](bool force) -> bool {
        if (pend == 1) {
            if (force) {
                if (!warp_wait(bar(B_DUMPED), pe_e & 1, p.status)) return false;
            } else if (!test_bar(B_DUMPED, pe_e & 1)) {
                return true;
            }
            if (!do_merge()) return false;
        }
        if (pend == 2) {
            if (force) {
                if (!warp_wait(bar(B_MERGED), pe_e & 1, p.status)) return false;
            } else if (!test_bar(B_MERGED, pe_e & 1)) {
                return true;
            }
            do_backproj();
        }
        return true;
    };
    auto segment_end = [&](const int32_t *h, uint32_t sbase, int seq) -> bool {
        // the previous end is complete for this warp, and every merge of it has
        // read the dumps: the dump area is free
        if (!poll(true)) return false;
        const int nvt = h[H_PV_RV8] / 8;
        const float lq = quad_sum(l_w);
        if (act) {
#pragma unroll
            for (int x = 0; x < kMaxNt; ++x)
                if (x < nvt) myregion[x * 32 + lane] = make_float2(vacc[x][0] + vacc[x][2], vacc[x][1] + vacc[x][3]);
        }
        myregion[kMaxNt * 32 + lane] = make_float2(act ? m_w : -INFINITY, act ? lq : 0.f);
        reset_state();
        arrive(B_QFREE + cur_b);  // the segment's q~ buffer is no longer read by this warp
        arrive(B_DUMPED);
        pend = 1;
        pe_e = nends++;
        pe_seq = seq;
        pe_pv = sbase + h[H_PV_OFF];
        pe_g = h[H_PV_G];
        pe_rg = h[H_PV_PASS] * ngrp + grp;
        pe_rv8 = h[H_PV_RV8];
        pe_run = h[H_PV_RUN];
        pe_rec = h[H_PV_REC];
        return true;
    };

    // ---- P^K part: this warp's slice of q~ for a coming segment
    auto project = [&](const int32_t *f, uint32_t sbase) -> bool {
        const int j = f[0], g = f[1], rk8 = f[2];
        const int rg = f[3] * ngrp + grp;
        const uint32_t pk = sbase + f[4];
        const int b = j & 1, u = j >> 1;
        // the buffer is free once every warp has ended segment j - 2
        if (u >= 1 && !warp_wait(bar(B_QFREE + b), (u - 1) & 1, p.status)) return false;
        if (rg < p.nrg) {
            uint32_t *qs = qs_part(b);
            const int rho = 8 * rg + quad;
            const uint16_t *qrow = nullptr;
            if (rho < p.rows_g) qrow = qsrc + ((int64_t)(rho / p.G) * p.hq + g * p.G + rho % p.G) * D;
            uint32_t qa[kMaxKs], qb[kMaxKs];
#pragma unroll
            for (int kc = 0; kc < kMaxKs; ++kc) {
                qa[kc] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 2 * qlane) : 0u;
                qb[kc] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 8 + 2 * qlane) : 0u;
            }
            const int njt = 2 * ((rk8 + 15) / 16);
            // rank tiles wi, wi + nwg, ... with two accumulators each (even / odd k-steps);
            // a rolled loop: this code runs a few times per launch, mostly from a cold
            // instruction cache, so its size matters more than its ILP
#pragma unroll 1
            for (int jt = wi; jt < njt; jt += nwg) {
                {
                    float acc0[4] = {0.f, 0.f, 0.f, 0.f}, acc1[4] = {0.f, 0.f, 0.f, 0.f};
                    if (jt < rk8 / 8) {
#pragma unroll
                        for (int kc = 0; kc < kMaxKs; kc += 2) {
                            // cores (jt, 2kc .. 2kc+3) of P^K: k-steps kc and kc+1
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4(pk + (jt * (D / 8) + 2 * kc + mi) * 128 + (lane % 8) * 16, b0, b1, b2, b3);
                            const uint32_t a0[4] = {qa[kc], 0u, qb[kc], 0u};
                            const uint32_t a1[4] = {qa[kc + 1], 0u, qb[kc + 1], 0u};
                            mma16816(acc0, a0, b0, b1);
                            mma16816(acc1, a1, b2, b3);
                        }
                    }
                    uint32_t hi, lo;
                    split_hi_lo((acc0[0] + acc1[0]) * p.scale_log2, (acc0[1] + acc1[1]) * p.scale_log2, hi, lo);
                    qs[((jt / 2) * 32 + lane) * 4 + (jt & 1) * 2 + 0] = hi;
                    qs[((jt / 2) * 32 + lane) * 4 + (jt & 1) * 2 + 1] = lo;
                }
            }
        }
        arrive(B_QREADY + b);
        return true;
    };

    // ---- start of a segment (one row-group pass of it): its q~ is in buffer j & 1
    auto segment_start = [&](const int32_t *h) -> bool {
        const int j = h[H_SS_J];
        const int b = j & 1, u = j >> 1;
        if (!warp_wait(bar(B_QREADY + b), u & 1, p.status)) return false;
        act = h[H_SS_PASS] * ngrp + grp < p.nrg;
        cur_b = b;
        reset_state();
        return true;
    };

    // Tile addressing shared by coefficient tiles and tail items (one copy of the
    // tile code): 128-byte cores from t_k / t_v, core (token group tg, rank
    // group rg) at tg * t_tgs + rg * t_rgs cores (coefficients: token-group
    // major; tail items: column-group major), t_ntg token groups valid.
    uint32_t t_k = 0, t_v = 0;
    int t_tgk = 1, t_rgk = 1, t_tgv = 1, t_rgv = 1, t_ntg = 4, t_nrk = 0, t_nrv = 0;
    auto kaddr = [&](int hf, int m4, int kk) -> uint32_t {
        const int tg = 2 * hf + (m4 >> 1), rgk = 2 * kk + (m4 & 1);
        return (tg < t_ntg && rgk < t_nrk) ? t_k + (tg * t_tgk + rgk * t_rgk) * 128 + (lane % 8) * 16 : zero_addr;
    };
    auto vaddr = [&](int hf, int m4, int jp) -> uint32_t {
        const int tg = 2 * hf + (m4 & 1), rgv = 2 * jp + (m4 >> 1);
        return (tg < t_ntg && rgv < t_nrv) ? t_v + (tg * t_tgv + rgv * t_rgv) * 128 + (lane % 8) * 16 : zero_addr;
    };
    auto run_tile = [&](float sc_mul, int tok_base, int t1) {
        by_width(max((t_nrk + 1) / 2, (t_nrv + 1) / 2),
                 [&](auto nkc) { tile32(nkc, sc_mul, tok_base, t1, t_ntg, kaddr, vaddr); });
    };

    // ---- tiles of one fill: the coefficient tiles this warp takes, or the whole
    // tail item when this warp owns one of its row groups.  One call site of the
    // tile code for both.
    auto fill_tiles = [&](const int32_t *h, uint32_t sbase, int flags) -> bool {
        int njobs = 0, kt0 = 0, ntl = 0, last8 = 0, t0 = 0, t1 = 0, rk8 = 0, rv8 = 0, rgt = -1;
        uint32_t kbase = 0, vbase = 0;
        float sc_mul = 1.f;
        if (flags & kHasC) {
            t0 = h[H_T0];
            t1 = h[H_T1];
            const int tok8 = h[H_TOK8];
            rk8 = h[H_RK8];
            rv8 = h[H_RV8];
            ntl = (t1 - t0 + kTileTokens - 1) / kTileTokens;
            if (act) {
                last8 = tok8 - (ntl - 1) * kTileTokens;
                kbase = sbase + h[H_C_OFF];
                vbase = kbase + tok8 * rk8 * 2;
                kt0 = (wi - tile_base % nwg + nwg) % nwg;  // this warp's first tile in the fill
                a_frag = smem_u32(qs_part(cur_b));
                njobs = kt0 < ntl ? (ntl - kt0 + nwg - 1) / nwg : 0;
                t_nrk = rk8 / 8;
                t_nrv = rv8 / 8;
                t_tgk = t_nrk;
                t_tgv = t_nrv;
                t_rgk = t_rgv = 1;
            }
            tile_base += ntl;
        } else if (flags & kTailFill) {
            for (int r = 0; r < p.nrg_t; ++r)
                if ((tail_ctr + r) % kMmaWarps == mw) rgt = r;
            tail_ctr += p.nrg_t;
            if (rgt >= 0) {
                const int i = h[H_QI], g = h[H_G];
                t1 = h[H_T1] - h[H_T0];  // tokens of the item
                reset_state();
                // tails come after the prefix: once the last segment end is through, no
                // warp reads this warp's dump area again; stage the item's A fragments there
                if (!poll(true)) return false;
                const int rloc = 8 * rgt + quad;  // query head within the KV group
                const uint16_t *qrow = (rloc < p.G) ? qsrc + ((int64_t)i * p.hq + g * p.G + rloc) * D : nullptr;
                uint32_t *fr = reinterpret_cast<uint32_t *>(myregion);
#pragma unroll 1
                for (int kk = 0; kk < kMaxKs; ++kk) {
                    float2 x0 = make_float2(0.f, 0.f), x1 = make_float2(0.f, 0.f);
                    if (qrow) {
                        x0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(qrow + 16 * kk + 2 * qlane));
                        x1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(qrow + 16 * kk + 8 + 2 * qlane));
                    }
                    uint32_t h0, l0, h1, l1;
                    split_hi_lo(x0.x * p.scale_log2, x0.y * p.scale_log2, h0, l0);
                    split_hi_lo(x1.x * p.scale_log2, x1.y * p.scale_log2, h1, l1);
                    *reinterpret_cast<uint4 *>(fr + (kk * 32 + lane) * 4) = make_uint4(h0, l0, h1, l1);
                }
                __syncwarp();
                a_frag = smem_u32(myregion);
                // the item arrives as one coefficient-style tile of kTailTokens tokens and rank d
                kbase = sbase;
                vbase = sbase + (D / 8) * kTailTokens * 16;
                njobs = (t1 + kTileTokens - 1) / kTileTokens;
                t_nrk = t_nrv = kMaxNt;
                t_tgk = t_tgv = 1;
                t_rgk = t_rgv = kTailTokens / 8;
            }
        }
        for (int jb = 0; jb < njobs; ++jb) {
            int tok_base;
            if (rgt < 0) {
                const int kt = kt0 + jb * nwg;
                t_ntg = ((kt == ntl - 1) ? last8 : kTileTokens) / 8;
                t_k = kbase + kt * kTileTokens * rk8 * 2;
                t_v = vbase + kt * kTileTokens * rv8 * 2;
                tok_base = t0 + kt * kTileTokens;
            } else {
                t_ntg = 4;
                t_k = kbase + 4 * jb * 128;
                t_v = vbase + 4 * jb * 128;
                tok_base = kTileTokens * jb;
            }
            run_tile(sc_mul, tok_base, t1);
        }
        if (rgt >= 0) {
            const int item = h[H_ITEM];
            float *rec = p.rec + (p.tail_rec_base + (int64_t)item * p.nrg_t + rgt) * recf;
#pragma unroll
            for (int x = 0; x < kMaxNt; ++x)
                __stcg(reinterpret_cast<float2 *>(rec + quad * D + 8 * x + 2 * qlane),
                       make_float2(vacc[x][0] + vacc[x][2], vacc[x][1] + vacc[x][3]));
            const float lq = quad_sum(l_w);
            if (qlane == 0) {
                __stcg(rec + 8 * D + quad, m_w);
                __stcg(rec + 8 * D + 8 + quad, lq);
            }
        }
        return true;
    };

    pdl_wait();  // q and the records belong to the preceding grids until here
    if (qcached) {  // q is 4-byte aligned (checked on the host)
        const int n4 = (int)((int64_t)p.batch * p.hq * D * 2 / 4);
        const uint32_t *src = reinterpret_cast<const uint32_t *>(p.q);
        uint32_t *dst = reinterpret_cast<uint32_t *>(smem + L::kQc);
        for (int k = mw * 32 + lane; k < n4; k += kMmaWarps * 32) dst[k] = src[k];
        if (!gsync()) return false;
    }
    for (int seq = 0;; ++seq) {
        const int slot = seq % kSlots;
        // the ring is about to come back to the fill still held for a back-projection
        if (pend != 0 && pe_seq % kSlots == slot && !poll(true)) return false;
        if (!warp_wait(bar(slot), (seq / kSlots) & 1, p.status)) return false;
        const int32_t *h = hdr + slot * kHdrInts;
        const int flags = h[H_FLAGS];
        const uint32_t sbase = smem_u32(smem + L::kRing + slot * kSlotBytes);
        if ((flags & kHasPv) && !segment_end(h, sbase, seq)) return false;
        if ((flags & kHasPk0) && !project(h + H_PK_J, sbase)) return false;
        if ((flags & kHasPk1) && !project(h + H_PK1_J, sbase)) return false;
        if ((flags & kSegStart) && !segment_start(h)) return false;
        if ((flags & (kHasC | kTailFill)) && !fill_tiles(h, sbase, flags)) return false;
        if (!(flags & kHasPv)) arrive(kSlots + slot);  // a fill with P^V is released by its back-projection
        if (flags & kEndFill) {
            if (!poll(true)) return false;
            break;
        }
        if (!poll(false)) return false;
    }
    return true;
}

// ================================================================ kernel
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    decode_kernel(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_v)
{
    using L = Lay<D>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    int32_t *hdr = reinterpret_cast<int32_t *>(smem + L::kHdr);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L::kBar);
    const uint32_t zero_addr = smem_u32(smem + L::kZero);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    pdl_trigger();
    if (threadIdx.x == 0) {
        for (int s = 0; s < kSlots; ++s) {
            mbar_init(smem_u32(&bars[s]), 1);                    // full: producer + bytes
            mbar_init(smem_u32(&bars[kSlots + s]), kMmaWarps);   // empty: every MMA warp
        }
        mbar_init(smem_u32(&bars[B_GS]), kMmaWarps);
        for (int b = B_QREADY; b < B_COUNT; ++b) mbar_init(smem_u32(&bars[b]), kMmaWarps);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x < 32) reinterpret_cast<uint32_t *>(smem + L::kZero)[threadIdx.x] = 0u;
    // dumps, q~ and merged v~ fragments: padding entries are read (times zero) before
    // they are first written, so they start as zeros
    for (int k = threadIdx.x; k < (L::kHdr - L::kMerge) / 4; k += kThreads)
        reinterpret_cast<uint32_t *>(smem + L::kMerge)[k] = 0u;
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) run_producer<D>(p, smem, hdr, bars, &tmap_k, &tmap_v);
    } else {
        run_mma<D>(p, smem, hdr, bars, zero_addr, warp - 1, lane);
    }
}


// ================================================================ combine
// The log-sum-exp merge of the split softmax (Eq. 1 over a partition of the
// tokens): one thread block per (KV head g, row group rg, float4 column c of
// the head dimension), one warp per row.  Lane l of a warp takes source
// records l, l + 32, ...; its loads are all in flight at once, and the 32
// partial merges meet through a shuffle butterfly.
template <int D>
__global__ void __launch_bounds__(256) combine_kernel(const __grid_constant__ DecodeParams p)
{
    constexpr int kC4 = D / 4;    // float4 columns of a row
    constexpr int kChunk = 8;     // records in flight per lane and round
    pdl_trigger();
    pdl_wait();  // every record of the decode grid is written
    const int c4 = blockIdx.x % kC4, rg = (blockIdx.x / kC4) % p.nrg, g = blockIdx.x / (kC4 * p.nrg);
    const int k = threadIdx.x / 32, sl = threadIdx.x % 32;
    const int recf = 8 * D + kRecFloatsExtra;
    const int rho = 8 * rg + k;
    const bool row_ok = rho < p.rows_g;
    const int i = row_ok ? rho / p.G : 0, hh = row_ok ? rho % p.G : 0;
    const int gs0 = p.g_slot_begin[g], nprefix = p.g_slot_begin[g + 1] - gs0;
    const int S = p.tail_splits, nsrc = row_ok ? nprefix + S : 0;
    const float *tail0 = p.rec + (p.tail_rec_base + (int64_t)(i * p.hkv + g) * S * p.nrg_t + hh / 8) * recf;
    float M = -INFINITY, Lsum = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s0 = sl; s0 < nsrc; s0 += kChunk * 32) {
        float mm[kChunk], ll[kChunk];
        float4 oo[kChunk];
#pragma unroll
        for (int j = 0; j < kChunk; ++j) {
            const int s = s0 + j * 32;
            mm[j] = -INFINITY;
            ll[j] = 0.f;
            oo[j] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (s < nsrc) {
                const bool pre = s < nprefix;
                const int row = pre ? k : hh % 8;
                const float *r = pre ? p.rec + ((int64_t)(gs0 + s) * p.nrg + rg) * recf
                                     : tail0 + (int64_t)(s - nprefix) * p.nrg_t * recf;
                mm[j] = __ldcg(r + 8 * D + row);
                ll[j] = __ldcg(r + 8 * D + 8 + row);
                oo[j] = __ldcg(reinterpret_cast<const float4 *>(r + row * D) + c4);
            }
        }
        float Mc = M;
#pragma unroll
        for (int j = 0; j < kChunk; ++j) Mc = fmaxf(Mc, mm[j]);
        const float a = exp2_diff(M, Mc);
        Lsum *= a;
        acc.x *= a; acc.y *= a; acc.z *= a; acc.w *= a;
#pragma unroll
        for (int j = 0; j < kChunk; ++j) {
            const float w = exp2_diff(mm[j], Mc);
            Lsum += w * ll[j];
            acc.x += w * oo[j].x; acc.y += w * oo[j].y; acc.z += w * oo[j].z; acc.w += w * oo[j].w;
        }
        M = Mc;
    }
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float Mo = __shfl_xor_sync(0xffffffffu, M, off);
        const float Lo = __shfl_xor_sync(0xffffffffu, Lsum, off);
        const float4 ao = make_float4(__shfl_xor_sync(0xffffffffu, acc.x, off), __shfl_xor_sync(0xffffffffu, acc.y, off),
                                      __shfl_xor_sync(0xffffffffu, acc.z, off), __shfl_xor_sync(0xffffffffu, acc.w, off));
        const float Mn = fmaxf(M, Mo);
        const float a = exp2_diff(M, Mn), b = exp2_diff(Mo, Mn);
        Lsum = Lsum * a + Lo * b;
        acc = make_float4(acc.x * a + ao.x * b, acc.y * a + ao.y * b, acc.z * a + ao.z * b, acc.w * a + ao.w * b);
        M = Mn;
    }
    if (row_ok && sl == 0) {
        const float inv = 1.f / Lsum;
        float *dst = p.out + ((int64_t)i * p.hq + g * p.G + hh) * D;
        reinterpret_cast<float4 *>(dst)[c4] = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
    }
}

}  // namespace

// Scratch of milo_attn_decode_static: the split-softmax partial records of
// one call live here instead of in a caller-provided workspace.  Every GPU
// that loads the library holds this array until the process exits.
static __device__ __align__(256) unsigned char g_static_workspace[kStaticWorkspaceBytes];

cudaError_t static_workspace(void **ptr)
{
    // Host code cannot use the array's name as a device address: look the
    // address up once per device, with that device current, and keep it.
    static std::mutex mu;
    static void *addr[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_workspace);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
    }
    *ptr = addr[dev];
    return cudaSuccess;
}

int decode_smem_bytes(int head_dim, int /*nrg_cta*/)
{
    return (head_dim == 64 ? Lay<64>::kTotal : Lay<128>::kTotal) + 1024;
}

cudaError_t launch_decode(const DecodeParams &p, const void *tmap_k, const void *tmap_v, int smem_bytes,
                          int num_ctas, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(num_ctas);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = (size_t)smem_bytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const CUtensorMap &mk = *static_cast<const CUtensorMap *>(tmap_k);
    const CUtensorMap &mv = *static_cast<const CUtensorMap *>(tmap_v);
    static int configured[kMaxDevices][2] = {};  // largest dynamic smem size set, per device and kernel
    const int which = p.d == 64 ? 0 : 1;
    const int dev = attribute_slot();
    if (p.num_chunks == 0 && (dev < 0 || smem_bytes > configured[dev][which])) {
        cudaError_t e = which == 0 ? cudaFuncSetAttribute(decode_kernel<64>,
                                                          cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes)
                                   : cudaFuncSetAttribute(decode_kernel<128>,
                                                          cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
        if (e != cudaSuccess) return e;
        if (dev >= 0) configured[dev][which] = smem_bytes;
    }
    cudaError_t e = p.num_chunks > 0 ? launch_chunks(p, tmap_k, tmap_v, stream)
                    : which == 0 ? cudaLaunchKernelEx(&cfg, decode_kernel<64>, p, mk, mv)
                                      : cudaLaunchKernelEx(&cfg, decode_kernel<128>, p, mk, mv);
    if (e != cudaSuccess || p.num_chunks > 0) return e;  // the short-block grid merges itself
    // the merge of the partial records, overlapping the decode grid's tail
    cudaLaunchConfig_t cc = cfg;
    cc.gridDim = dim3(p.hkv * p.nrg * (p.d / 4));
    cc.blockDim = dim3(256);
    cc.dynamicSmemBytes = 0;
    return which == 0 ? cudaLaunchKernelEx(&cc, combine_kernel<64>, p) : cudaLaunchKernelEx(&cc, combine_kernel<128>, p);
}

}  // namespace milo
