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
// One persistent thread block per SM with four warp roles:
//   producer    (warp 0, one lane): walks the block's static list of prefix
//               segments, bulk-copies each segment's P^K and P^V into their
//               own buffers (P^V double-buffered) and its packed coefficient tiles into a ring of
//               slots (1-D cp.async.bulk, mbarrier completion); grabs dense
//               tail items from a counter and streams them with 3-D TMA.
//   projection  (warp 1): q~ = scale * log2(e) * P^K q for every segment, as
//               bf16 hi + lo mma fragments, into a shared buffer.
//   MMA warps   (warps 4..11): 16-token sub-tiles round-robin: scores (mma
//               m16n8k16; A rows 0-7 = q~ hi, 8-15 = q~ lo), online softmax
//               in registers, rank-space values (A rows = p hi / p lo).  At a
//               segment's end each warp dumps (max, sum, v~) into its own
//               shared-memory region and continues with the next segment.
//   epilogue    (warps 2-3): both merge the 8 dumps of a segment; each
//               back-projects v~ through P^V into half of the head dimension,
//               folds it into its half of the run's output and writes it to
//               the partial record; the first counts the tickets.
// The thread block that brings the last record of a (KV head, row group)
// merges all of that row group's records at the end of the kernel (no
// thread block ever waits for another).  Every wait is bounded (~2 s); on
// expiry the thread records MILO_ERR_TIMEOUT in the sticky status word and
// leaves.
#include <cuda.h>
#include <cuda_bf16.h>

#include <mutex>

#include "milo.h"
#include "milo_internal.h"

namespace milo {
namespace {

constexpr uint64_t kTimeoutNs = 2000000000ull;

enum : int { kEnd = 0, kC = 2, kTail = 4 };             // ring slot kinds
enum : int { kPkEnd = 0, kPkSeg = 1 };                  // P^K buffer kinds
enum : int { kDumpEnd = 0, kDumpSeg = 1, kDumpTail = 2 };
enum : int { F_FIRST_C = 1, F_LAST_C = 2, F_RUN_FIRST = 4, F_RUN_LAST = 8 };
// ring slot header words
enum : int { H_KIND, H_E, H_G, H_T0, H_T1, H_RK8, H_RV8, H_TOK8, H_NSUB, H_FLAGS, H_REC, H_PASS, H_QI, H_ITEM };
// barrier indices (after the ring's full[kSlots], empty[kSlots])
enum : int {
    B_PKF = 2 * kSlots, B_PKE, B_PVF0, B_PVF1, B_PVE0, B_PVE1, B_QR, B_QF, B_MF, B_ME, B_EPS, B_FIN, B_COUNT
};

// ------------------------------------------------------------------ PTX ----
__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t tx)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(tx) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: false (and the status word set) once kTimeoutNs has passed.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int32_t *status)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 32; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer() - t0 > kTimeoutNs) {
            atomicCAS(status, 0, (int32_t)MILO_ERR_TIMEOUT);
            return false;
        }
    }
}

// Warp-uniform bounded wait: every lane waits; all agree on the outcome.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, int32_t *status)
{
    const bool ok = mbar_wait(bar, parity, status);
    return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int c0, int c1, int c2,
                                            uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(map), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D(16x8 f32) += A(16x16 bf16, row) * B(16x8 bf16, col)
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" :::); }

// Two floats -> bf16x2 (low half = first) rounded to nearest, and the
// bf16x2 of their rounding residuals: x = hi + lo to ~16 significant bits.
__device__ __forceinline__ void split_hi_lo(float x0, float x1, uint32_t &hi, uint32_t &lo)
{
    const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

__device__ __forceinline__ float quad_max(float v)
{
    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
    return fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
}

__device__ __forceinline__ float quad_sum(float v)
{
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    return v + __shfl_xor_sync(0xffffffffu, v, 2);
}

// exp2(a - b) with the convention that a = -inf gives 0 (and b = -inf too).
__device__ __forceinline__ float exp2_diff(float a, float b)
{
    return (a == -INFINITY) ? 0.f : exp2f(a - b);
}

// ------------------------------------------------------- shared memory ----
template <int D>
struct Lay {
    static constexpr int al(int x, int a) { return (x + a - 1) / a * a; }
    static constexpr int kPBytes = D * D * 2;                   // largest P (r <= d)
    static constexpr int kPk = kSlots * kSlotBytes;             // ring at 0
    static constexpr int kPv = kPk + kPBytes;                   // two P^V buffers
    static constexpr int kMerge = kPv + 2 * kPBytes;
    static constexpr int kMergeWarp = 32 * D + 256;             // v~ [d/8][32 lanes] float2 + (m,l) [32] float2
    static constexpr int kQsPart = (D / 16) * 32 * 16;          // q~ fragments of one row group
    static constexpr int kQs = kMerge + kMmaWarps * kMergeWarp;
    static constexpr int kHdr = kQs + 2 * kQsPart;              // ring headers, P^K header, dump descriptor
    static constexpr int kBar = al(kHdr + (kSlots + 2) * 64, 128);
    static constexpr int kZero = al(kBar + B_COUNT * 8, 128);
    static constexpr int kList = kZero + 128;                   // deferred combines: count, (g, rg) pairs
    static constexpr int kListCap = 255;
    static constexpr int kTotal = kList + 8 * (kListCap + 1);
    static_assert(kPk % 1024 == 0 && kSlotBytes % 1024 == 0, "ring alignment (128B-swizzled TMA boxes)");
    static_assert(kPv % 128 == 0 && kMerge % 128 == 0 && kQs % 128 == 0 && kHdr % 128 == 0, "alignment");
    static_assert(kZero % 128 == 0, "zero line alignment");
    static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// ------------------------------------------------------- combine ----------
// Merge every partial record of (KV head g, row group rg) and write out.
template <int D>
__device__ void combine_rows(const DecodeParams &p, int g, int rg, int tid, int nthr)
{
    constexpr int kChunk = 12;  // records whose loads are in flight together
    const int recf = 8 * D + kRecFloatsExtra;
    const int gs0 = p.g_slot_begin[g], gs1 = p.g_slot_begin[g + 1];
    const int nprefix = gs1 - gs0;
    const int S = p.tail_splits;
    const int nsrc = nprefix + S;
    for (int w = tid; w < 8 * (D / 4); w += nthr) {
        const int k = w / (D / 4), c4 = w % (D / 4);
        const int rho = 8 * rg + k;
        if (rho >= p.rows_g) continue;
        const int i = rho / p.G, hh = rho % p.G;
        const float *tail0 = p.rec + (p.tail_rec_base + (int64_t)(i * p.hkv + g) * S * p.nrg_t + hh / 8) * recf;
        float M = -INFINITY, Lsum = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s0 = 0; s0 < nsrc; s0 += kChunk) {
            float mm[kChunk], ll[kChunk];
            float4 oo[kChunk];
#pragma unroll
            for (int j = 0; j < kChunk; ++j) {
                const int s = s0 + j;
                if (s < nsrc) {
                    const bool pre = s < nprefix;
                    const int row = pre ? k : hh % 8;
                    const float *r = pre ? p.rec + (int64_t)((gs0 + s) * p.nrg + rg) * recf
                                         : tail0 + (int64_t)(s - nprefix) * p.nrg_t * recf;
                    mm[j] = __ldcg(r + 8 * D + row);
                    ll[j] = __ldcg(r + 8 * D + 8 + row);
                    oo[j] = __ldcg(reinterpret_cast<const float4 *>(r + row * D) + c4);
                } else {
                    mm[j] = -INFINITY;
                    ll[j] = 0.f;
                    oo[j] = make_float4(0.f, 0.f, 0.f, 0.f);
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
                const float w8 = exp2_diff(mm[j], Mc);
                Lsum += w8 * ll[j];
                acc.x += w8 * oo[j].x;
                acc.y += w8 * oo[j].y;
                acc.z += w8 * oo[j].z;
                acc.w += w8 * oo[j].w;
            }
            M = Mc;
        }
        const float inv = 1.f / Lsum;
        float *dst = p.out + ((int64_t)i * p.hq + g * p.G + hh) * D;
        reinterpret_cast<float4 *>(dst)[c4] = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
    }
}

// Expected number of records for (g, rg): prefix runs of g plus tail items
// whose query rows meet the row group.
__device__ __forceinline__ int expected_arrivals(const DecodeParams &p, int g, int rg)
{
    int cnt = p.g_slot_begin[g + 1] - p.g_slot_begin[g];
    if (p.tail_splits > 0) {
        const int r0 = 8 * rg, r1 = min(8 * rg + 8, p.rows_g);  // [r0, r1)
        const int i0 = r0 / p.G, i1 = (r1 - 1) / p.G;
        for (int i = i0; i <= i1; ++i)
            for (int t = 0; t < p.nrg_t; ++t) {
                const int a = i * p.G + 8 * t, b = i * p.G + min(8 * t + 8, p.G);
                if (a < r1 && b > r0) cnt += p.tail_splits;
            }
    }
    return cnt;
}

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
__device__ void run_producer(const DecodeParams &p, uint8_t *smem, int32_t *hdr, int32_t *pkh, uint64_t *bars,
                             const CUtensorMap *tmap_k, const CUtensorMap *tmap_v)
{
    using L = Lay<D>;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    int seq = 0, npk = 0, npv = 0;
    bool ok = true, waited = false;

    auto ring_acquire = [&]() -> int {
        const int slot = seq % kSlots;
        if (seq >= kSlots && !mbar_wait(bar(kSlots + slot), ((seq / kSlots) - 1) & 1, p.status)) return -1;
        return slot;
    };
    auto emit_pk = [&](int kind, int g, int rk8, int pass, int64_t off) -> bool {
        if (npk >= 1 && !mbar_wait(bar(B_PKE), (npk - 1) & 1, p.status)) return false;
        pkh[0] = kind;
        pkh[1] = g;
        pkh[2] = rk8;
        pkh[3] = pass;
        const uint32_t bytes = kind == kPkSeg ? (uint32_t)rk8 * D * 2 : 0u;
        if (bytes) {
            mbar_arrive_tx(bar(B_PKF), bytes);
            bulk_g2s(smem_u32(smem + L::kPk), p.packed + off, bytes, bar(B_PKF));
        } else {
            mbar_arrive(bar(B_PKF));
        }
        ++npk;
        return true;
    };
    auto emit_pv = [&](int rv8, int64_t off) -> bool {
        const int b = npv & 1;  // double-buffered: the epilogue may still hold the other one
        if (npv >= 2 && !mbar_wait(bar(B_PVE0 + b), ((npv / 2) - 1) & 1, p.status)) return false;
        const uint32_t bytes = (uint32_t)rv8 * D * 2;
        if (bytes) {
            mbar_arrive_tx(bar(B_PVF0 + b), bytes);
            bulk_g2s(smem_u32(smem + L::kPv + b * L::kPBytes), p.packed + off, bytes, bar(B_PVF0 + b));
        } else {
            mbar_arrive(bar(B_PVF0 + b));
        }
        ++npv;
        return true;
    };
    auto emit_tail = [&](uint32_t item) -> bool {
        const int S = p.tail_splits;
        const int i = item / (p.hkv * S), g = (item / S) % p.hkv, sp = item % S;
        const int64_t o0 = p.tail_offsets[i], o1 = p.tail_offsets[i + 1];
        const int T = (int)(o1 - o0);
        if (sp == S - 1 && T > S * kTailTokens) atomicCAS(p.status, 0, (int32_t)MILO_ERR_DEVICE_BOUNDS);
        const int t0 = sp * kTailTokens, t1 = min(t0 + kTailTokens, T);
        for (int pass = 0; pass < p.npass_t; ++pass) {
            const int slot = ring_acquire();
            if (slot < 0) return false;
            int32_t *h = hdr + slot * kHdrInts;
            h[H_KIND] = kTail;
            h[H_G] = g;
            h[H_QI] = i;
            h[H_ITEM] = (int)item;
            h[H_T0] = t0;
            h[H_T1] = t1;
            h[H_PASS] = pass;
            h[H_RV8] = D;
            h[H_FLAGS] = 0;
            const uint32_t fb = bar(slot);
            if (t1 > t0) {
                constexpr uint32_t half = kTailTokens * 128;  // one box: kTailTokens rows x 64 columns
                constexpr uint32_t bytes = 2 * (D / 64) * half;
                mbar_arrive_tx(fb, bytes);
                const uint32_t dst = smem_u32(smem + slot * kSlotBytes);
                const int row = (int)(o0 + t0);
#pragma unroll
                for (int hb = 0; hb < D / 64; ++hb) {
                    tma_load_3d(dst + hb * half, tmap_k, 64 * hb, g, row, fb);
                    tma_load_3d(dst + (D / 64) * half + hb * half, tmap_v, 64 * hb, g, row, fb);
                }
            } else {
                mbar_arrive(fb);
            }
            ++seq;
        }
        return true;
    };
    const uint32_t tail_quota =
        p.has_tail ? (uint32_t)((p.num_tail_items + p.num_ctas - 1) / p.num_ctas) : 0u;
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
    bool first_segment = true;
    if (!it.done) {
        const SegDev s0 = p.segs[it.sg];
        const EntryDev e0 = p.entries[s0.entry];
        ok = emit_pk(kPkSeg, e0.g, (e0.rk + 7) & ~7, it.pass, e0.off_pk);
    }
    while (ok && !it.done) {
        const SegDev seg = p.segs[it.sg];
        const EntryDev ent = p.entries[seg.entry];
        const int rk8 = (ent.rk + 7) & ~7, rv8 = (ent.rv + 7) & ~7;
        int runfl = 0;
        if (it.sg == it.r0) runfl |= F_RUN_FIRST;
        if (it.sg == it.r1) runfl |= F_RUN_LAST;
        SegIter nx = it;
        nx.advance(p);
        bool pk_next = nx.done;
        const int per_tile = kTileTokens * (rk8 + rv8) * 2;
        int tps = per_tile > 0 ? kSlotBytes / per_tile : 16;
        tps = max(1, min(tps, 16));
        const int n8 = (ent.n + 7) & ~7;
        const int nsl = (seg.t1 - seg.t0 + tps * kTileTokens - 1) / (tps * kTileTokens);
        const int pk_at = first_segment ? min(kSlots - 1, nsl - 1) : min(1, nsl - 1);
        for (int si = 0; si < nsl && ok; ++si) {
            const int tt0 = seg.t0 + si * tps * kTileTokens;
            const int tt1 = min(seg.t1, tt0 + tps * kTileTokens);
            const int tok8 = min((tt1 + 7) & ~7, n8) - tt0;
            const int ntl = (tt1 - tt0 + kTileTokens - 1) / kTileTokens;
            const int last8 = tok8 - (ntl - 1) * kTileTokens;
            const int nsub = 2 * (ntl - 1) + (last8 + 15) / 16;
            const int slot = ring_acquire();
            if (slot < 0) { ok = false; break; }
            int32_t *h = hdr + slot * kHdrInts;
            h[H_KIND] = kC;
            h[H_E] = seg.entry;
            h[H_G] = ent.g;
            h[H_T0] = tt0;
            h[H_T1] = tt1;
            h[H_RK8] = rk8;
            h[H_RV8] = rv8;
            h[H_TOK8] = tok8;
            h[H_NSUB] = nsub;
            h[H_FLAGS] = runfl | (si == 0 ? F_FIRST_C : 0) | (si == nsl - 1 ? F_LAST_C : 0);
            h[H_REC] = seg.slot;
            h[H_PASS] = it.pass;
            const uint32_t kb = (uint32_t)tok8 * rk8 * 2, vb = (uint32_t)tok8 * rv8 * 2;
            const uint32_t fb = bar(slot);
            if (kb + vb) {
                mbar_arrive_tx(fb, kb + vb);
                const uint32_t dst = smem_u32(smem + slot * kSlotBytes);
                if (kb) bulk_g2s(dst, p.packed + ent.off_ck + (int64_t)tt0 * rk8 * 2, kb, fb);
                if (vb) bulk_g2s(dst + kb, p.packed + ent.off_cv + (int64_t)tt0 * rv8 * 2, vb, fb);
            } else {
                mbar_arrive(fb);
            }
            ++seq;
            if (!pk_next && si == pk_at) {
                // the next segment's basis, early, so its q~ is ready in time
                const SegDev ns = p.segs[nx.sg];
                const EntryDev ne = p.entries[ns.entry];
                ok = emit_pk(kPkSeg, ne.g, (ne.rk + 7) & ~7, nx.pass, ne.off_pk);
                pk_next = true;
            }
        }
        if (!ok) break;
        ok = emit_pv(rv8, ent.off_pv);
        if (ok && first_segment) {
            pdl_wait();
            waited = true;
            ok = grab_tails(tail_quota);
        }
        first_segment = false;
        it = nx;
    }
    if (!waited) pdl_wait();
    if (ok) ok = grab_tails(0xffffffffu);
    if (ok) {
        const int slot = ring_acquire();
        if (slot >= 0) {
            hdr[slot * kHdrInts + H_KIND] = kEnd;
            mbar_arrive(bar(slot));
            ++seq;
        }
        emit_pk(kPkEnd, 0, 0, 0, 0);
    }
    // the last thread block to finish grabbing resets the tail counter
    if (atomicAdd(&p.counters->ctas_done, 1u) == (uint32_t)p.num_ctas - 1) {
        p.counters->tail_next = 0u;
        p.counters->ctas_done = 0u;
    }
    // do not leave while a copy this thread started may still be landing
    for (int j = max(0, seq - kSlots); j < seq; ++j)
        if (!mbar_wait(bar(j % kSlots), (j / kSlots) & 1, p.status)) break;
    if (npk > 0) mbar_wait(bar(B_PKF), (npk - 1) & 1, p.status);
    for (int j = max(0, npv - 2); j < npv; ++j) mbar_wait(bar(B_PVF0 + (j & 1)), (j / 2) & 1, p.status);
}

// ================================================================ projection
template <int D>
__device__ bool run_projection(const DecodeParams &p, uint8_t *smem, const int32_t *pkh, uint64_t *bars, int lane)
{
    using L = Lay<D>;
    constexpr int kMaxKs = D / 16;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    const int quad = lane / 4, qlane = lane % 4;
    const uint32_t pk = smem_u32(smem + L::kPk);
    pdl_wait();
    for (int k = 0;; ++k) {
        if (!warp_wait(bar(B_PKF), k & 1, p.status)) return false;
        const int kind = pkh[0];
        if (kind == kPkEnd) return true;
        const int g = pkh[1], rk8 = pkh[2], pass = pkh[3];
        // the MMA warps load segment k-1's q~ when they start it, long before
        // segment k's basis arrives: one buffer suffices
        if (k >= 1 && !warp_wait(bar(B_QF), (k - 1) & 1, p.status)) return false;
        for (int grp = 0; grp < p.nrg_cta; ++grp) {
            const int rg = pass * p.nrg_cta + grp;
            const int rho = 8 * rg + quad;
            const uint16_t *qrow = nullptr;
            if (rg < p.nrg && rho < p.rows_g) {
                const int i = rho / p.G, hh = rho % p.G;
                qrow = p.q + ((int64_t)i * p.hq + g * p.G + hh) * D;
            }
            uint32_t qlo[kMaxKs], qhi[kMaxKs];
#pragma unroll
            for (int kc = 0; kc < kMaxKs; ++kc) {
                qlo[kc] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 2 * qlane) : 0u;
                qhi[kc] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 8 + 2 * qlane) : 0u;
            }
            uint4 *qs = reinterpret_cast<uint4 *>(smem + L::kQs + grp * L::kQsPart);
            const int njt = 2 * ((rk8 + 15) / 16);
            for (int jt = 0; jt < njt; ++jt) {
                float acc[4] = {0.f, 0.f, 0.f, 0.f};
                if (jt < rk8 / 8) {
#pragma unroll
                    for (int kc = 0; kc < kMaxKs; kc += 2) {
                        uint32_t b0, b1, b2, b3;
                        // tiles (jt, 2kc), (jt, 2kc+1), (jt, 2kc+2), (jt, 2kc+3) of P^K
                        const int cg = 2 * kc + (lane / 8);
                        ldsm_x4(pk + (jt * (D / 8) + cg) * 128 + (lane % 8) * 16, b0, b1, b2, b3);
                        const uint32_t a0[4] = {qlo[kc], 0u, qhi[kc], 0u};
                        const uint32_t a1[4] = {qlo[kc + 1], 0u, qhi[kc + 1], 0u};
                        mma16816(acc, a0, b0, b1);
                        mma16816(acc, a1, b2, b3);
                    }
                }
                uint32_t hi, lo;
                split_hi_lo(acc[0] * p.scale_log2, acc[1] * p.scale_log2, hi, lo);
                uint32_t *dst = reinterpret_cast<uint32_t *>(qs + (jt / 2) * 32 + lane);
                dst[(jt & 1) * 2 + 0] = hi;
                dst[(jt & 1) * 2 + 1] = lo;
            }
        }
        __syncwarp();
        if (lane == 0) {
            mbar_arrive(bar(B_PKE));
            mbar_arrive(bar(B_QR));
        }
    }
}

// ================================================================ MMA warps
template <int D>
__device__ bool run_mma(const DecodeParams &p, uint8_t *smem, const int32_t *hdr, int32_t *dsc, uint64_t *bars,
                        uint32_t zero_addr, int mw, int lane)
{
    using L = Lay<D>;
    constexpr int kMaxNt = D / 8;   // max rank (or column) 8-tiles
    constexpr int kMaxKs = D / 16;  // max 16-wide k-steps
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    const int quad = lane / 4, qlane = lane % 4;
    float2 *region = reinterpret_cast<float2 *>(smem + L::kMerge + mw * L::kMergeWarp);

    uint32_t qf[kMaxKs][4];
    float vacc[kMaxNt][4];
    float m_w = -INFINITY, l_w = 0.f;
    int nseg = 0, ndump = 0, sub_base = 0;
    bool active = false;

    pdl_wait();

    auto reset_state = [&]() {
        m_w = -INFINITY;
        l_w = 0.f;
#pragma unroll
        for (int x = 0; x < kMaxNt; ++x) vacc[x][0] = vacc[x][1] = vacc[x][2] = vacc[x][3] = 0.f;
    };

    // One 16-token sub-tile: scores, online softmax, rank-space values.
    // Keys/values are read through `kaddr(mi, kk)` / `vaddr(mi, jp)`.
    auto subtile = [&](int nks, int njp, float sc_mul, int tok_base, int t1, bool tgb_ok, auto kaddr, auto vaddr) {
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
        const int mi = lane / 8;
#pragma unroll
        for (int kk = 0; kk < kMaxKs; ++kk) {
            if (kk < nks) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4(kaddr(mi, kk), b0, b1, b2, b3);
                mma16816(sa, qf[kk], b0, b1);
                mma16816(sb, qf[kk], b2, b3);
            }
        }
        const int tokA = tok_base + 2 * qlane;
        float s0 = (sa[0] + sa[2]) * sc_mul, s1 = (sa[1] + sa[3]) * sc_mul;
        float s2 = (sb[0] + sb[2]) * sc_mul, s3 = (sb[1] + sb[3]) * sc_mul;
        if (tokA >= t1) s0 = -INFINITY;
        if (tokA + 1 >= t1) s1 = -INFINITY;
        if (!tgb_ok || tokA + 8 >= t1) s2 = -INFINITY;
        if (!tgb_ok || tokA + 9 >= t1) s3 = -INFINITY;
        const float mx = quad_max(fmaxf(fmaxf(s0, s1), fmaxf(s2, s3)));
        if (mx > m_w + 8.f) {  // lazy rescale: p stays <= 2^8
            const float alpha = exp2_diff(m_w, mx);
            l_w *= alpha;
#pragma unroll
            for (int x = 0; x < kMaxNt; ++x) {
                vacc[x][0] *= alpha; vacc[x][1] *= alpha; vacc[x][2] *= alpha; vacc[x][3] *= alpha;
            }
            m_w = mx;
        }
        const float p0 = exp2f(s0 - m_w), p1 = exp2f(s1 - m_w);
        const float p2 = exp2f(s2 - m_w), p3 = exp2f(s3 - m_w);
        l_w += (p0 + p1) + (p2 + p3);
        uint32_t pa[4];
        split_hi_lo(p0, p1, pa[0], pa[1]);
        split_hi_lo(p2, p3, pa[2], pa[3]);
#pragma unroll
        for (int jp = 0; jp < kMaxKs; ++jp) {
            if (jp < njp) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vaddr(mi, jp), b0, b1, b2, b3);
                mma16816(vacc[2 * jp], pa, b0, b1);
                mma16816(vacc[2 * jp + 1], pa, b2, b3);
            }
        }
    };

    // Hand this warp's (max, sum, v~) to the epilogue warp.
    auto dump = [&](int kind, const int32_t *h, int nvt) -> bool {
        if (ndump >= 1 && !warp_wait(bar(B_ME), (ndump - 1) & 1, p.status)) return false;
        const float lq = quad_sum(l_w);
        if (active) {
#pragma unroll
            for (int x = 0; x < kMaxNt; ++x)
                if (x < nvt) region[x * 32 + lane] = make_float2(vacc[x][0] + vacc[x][2], vacc[x][1] + vacc[x][3]);
        }
        region[kMaxNt * 32 + lane] = make_float2(active ? m_w : -INFINITY, active ? lq : 0.f);
        if (mw == 0 && lane == 0) {
            dsc[0] = kind;
            if (h) {
                dsc[1] = h[H_G];
                dsc[2] = h[H_RV8];
                dsc[3] = h[H_FLAGS];
                dsc[4] = h[H_REC];
                dsc[5] = h[H_PASS];
                dsc[6] = h[H_ITEM];
                dsc[7] = h[H_QI];
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(B_MF));
        ++ndump;
        return true;
    };

    for (int seq = 0;; ++seq) {
        const int slot = seq % kSlots;
        if (!warp_wait(bar(slot), (seq / kSlots) & 1, p.status)) return false;
        const int32_t *h = hdr + slot * kHdrInts;
        const int kind = h[H_KIND];
        const uint32_t sbase = smem_u32(smem + slot * kSlotBytes);
        if (kind == kEnd) {
            active = false;
            if (!dump(kDumpEnd, nullptr, 0)) return false;
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kSlots + slot));
            return true;
        }
        if (kind == kC) {
            const int ngrp = p.nrg_cta, grp = mw % ngrp, phase = mw / ngrp, ts = kMmaWarps / ngrp;
            const int rg = h[H_PASS] * ngrp + grp;
            const int flags = h[H_FLAGS], rk8 = h[H_RK8], rv8 = h[H_RV8];
            const int nks = (rk8 + 15) / 16, njp = (rv8 + 15) / 16;
            if (flags & F_FIRST_C) {
                if (!warp_wait(bar(B_QR), nseg & 1, p.status)) return false;
                active = rg < p.nrg;
                if (active) {
                    const uint4 *qs = reinterpret_cast<const uint4 *>(smem + L::kQs + grp * L::kQsPart);
#pragma unroll
                    for (int kk = 0; kk < kMaxKs; ++kk)
                        if (kk < nks) {
                            const uint4 v = qs[kk * 32 + lane];
                            qf[kk][0] = v.x; qf[kk][1] = v.y; qf[kk][2] = v.z; qf[kk][3] = v.w;
                        }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(B_QF));
                reset_state();
                ++nseg;
            }
            if (active) {
                const int t0 = h[H_T0], t1 = h[H_T1], tok8 = h[H_TOK8], nsub = h[H_NSUB];
                const uint32_t kbase = sbase, vbase = sbase + tok8 * rk8 * 2;
                const int ntl = (t1 - t0 + kTileTokens - 1) / kTileTokens;
                for (int u = 0; u < nsub; ++u) {
                    if ((sub_base + u) % ts != phase) continue;
                    const int kt = u / 2, su = u % 2;
                    const int t8 = (kt == ntl - 1) ? tok8 - kt * kTileTokens : kTileTokens;
                    const int ntg = t8 / 8;
                    const int tga = 2 * su, tgb = tga + 1;
                    const uint32_t ktile = kbase + kt * kTileTokens * rk8 * 2;
                    const uint32_t vtile = vbase + kt * kTileTokens * rv8 * 2;
                    auto kaddr = [&](int mi, int kk) -> uint32_t {
                        const int tg = (mi < 2) ? tga : tgb, rgk = 2 * kk + (mi & 1);
                        return (tg < ntg && rgk < rk8 / 8) ? ktile + (rgk * ntg + tg) * 128 + (lane % 8) * 16
                                                           : zero_addr;
                    };
                    auto vaddr = [&](int mi, int jp) -> uint32_t {
                        const int tg = (mi & 1) ? tgb : tga, rgv = 2 * jp + (mi >> 1);
                        return (tg < ntg && rgv < rv8 / 8) ? vtile + (rgv * ntg + tg) * 128 + (lane % 8) * 16
                                                           : zero_addr;
                    };
                    subtile(nks, njp, 1.f, t0 + kt * kTileTokens + 8 * tga, t1, tgb < ntg, kaddr, vaddr);
                }
                sub_base += nsub;
            }
            if (flags & F_LAST_C)
                if (!dump(kDumpSeg, h, rv8 / 8)) return false;
        } else if (kind == kTail) {
            const int ngrp = p.ngrp_t, grp = mw % ngrp, phase = mw / ngrp, ts = kMmaWarps / ngrp;
            const int rgt = h[H_PASS] * ngrp + grp;
            active = rgt < p.nrg_t;
            reset_state();
            if (active) {
                const int i = h[H_QI], g = h[H_G], t0 = h[H_T0], t1 = h[H_T1];
                const int rloc = 8 * rgt + quad;  // query head within the KV group
                const uint16_t *qrow = (rloc < p.G) ? p.q + ((int64_t)i * p.hq + g * p.G + rloc) * D : nullptr;
#pragma unroll
                for (int kc = 0; kc < kMaxKs; ++kc) {
                    qf[kc][0] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 2 * qlane) : 0u;
                    qf[kc][1] = 0u;
                    qf[kc][2] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 8 + 2 * qlane) : 0u;
                    qf[kc][3] = 0u;
                }
                constexpr uint32_t half = kTailTokens * 128;
                const uint32_t kb = sbase, vb = sbase + (D / 64) * half;
                const int ntok = t1 - t0;
                const int nsub = (ntok + 15) / 16;
                for (int u = phase; u < nsub; u += ts) {
                    const int tga = 2 * u, tgb = tga + 1;
                    // 128B-swizzled boxes: row tr, 16-byte chunk ch at ((ch % 8) ^ (tr % 8))
                    auto kaddr = [&](int mi, int kc) -> uint32_t {
                        const int tr = 8 * ((mi < 2) ? tga : tgb) + (lane % 8), ch = 2 * kc + (mi & 1);
                        return kb + (ch / 8) * half + tr * 128 + (((ch % 8) ^ (tr % 8)) * 16);
                    };
                    auto vaddr = [&](int mi, int cp) -> uint32_t {
                        const int tr = 8 * ((mi & 1) ? tgb : tga) + (lane % 8), ch = 2 * cp + (mi >> 1);
                        return vb + (ch / 8) * half + tr * 128 + (((ch % 8) ^ (tr % 8)) * 16);
                    };
                    subtile(kMaxKs, kMaxKs, p.scale_log2, 8 * tga, ntok, true, kaddr, vaddr);
                }
            }
            if (!dump(kDumpTail, h, kMaxNt)) return false;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(kSlots + slot));
    }
}

// ================================================================ epilogue
template <int D>
__device__ bool run_epilogue(const DecodeParams &p, uint8_t *smem, const int32_t *dsc, uint64_t *bars,
                             int32_t *list, uint32_t zero_addr, int ep, int lane)
{
    using L = Lay<D>;
    constexpr int kMaxNt = D / 8;
    constexpr int kMaxKs = D / 16;
    constexpr int kHalf = kMaxNt / 2;      // column tiles of this warp's half of the head dimension
    const int ct0 = ep * kHalf;            // first column tile of this warp
    int neps = 0;                          // record hand-offs between the two epilogue warps
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    const int quad = lane / 4, qlane = lane % 4;
    const uint32_t pv_base = smem_u32(smem + L::kPv);
    const int recf = 8 * D + kRecFloatsExtra;
    auto region = [&](int w) { return reinterpret_cast<const float2 *>(smem + L::kMerge + w * L::kMergeWarp); };

    float orun[2][kHalf][2];
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
    int ndump = 0, npv = 0;
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int x = 0; x < kHalf; ++x) orun[a][x][0] = orun[a][x][1] = 0.f;
    // Both epilogue warps meet once their halves of a record are written (a
    // two-warp barrier: neither can run a phase ahead of the other); the
    // first one then counts the tickets.
    auto await_partner = [&]() -> bool {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(B_EPS));
        const bool ok = warp_wait(bar(B_EPS), neps & 1, p.status);
        ++neps;
        return ok;
    };

    pdl_wait();  // records and tickets belong to the preceding grid until here

    // Count one record of (g, rg).  The thread block bringing the last one
    // merges that row group: at the end of the kernel with every thread, or
    // right away with this warp when the deferral list is full.
    auto ticket = [&](int g, int rg) {
        int last = 0;
        if (lane == 0) {
            const uint32_t old = atomicAdd(&p.tickets[g * p.nrg + rg], 1u);
            last = (old == (uint32_t)expected_arrivals(p, g, rg) - 1) ? 1 : 0;
            if (last) {
                p.tickets[g * p.nrg + rg] = 0u;
                __threadfence();
            }
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (!last) return;
        if (list[0] < L::kListCap) {
            if (lane == 0) {
                const int n = list[0];
                list[1 + 2 * n] = g;
                list[2 + 2 * n] = rg;
                list[0] = n + 1;
            }
            __syncwarp();
        } else {
            combine_rows<D>(p, g, rg, lane, 32);
        }
    };

    // Merge weights of the warps of one row group: sc[w] = 2^(m_w - M).
    auto merge_scales = [&](int ngrp, int grp, float (&sc)[kMmaWarps], float &M, float &Lsum) {
        M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w)
            if (w % ngrp == grp) M = fmaxf(M, region(w)[kMaxNt * 32 + lane].x);
        Lsum = 0.f;
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w) {
            sc[w] = 0.f;
            if (w % ngrp == grp) {
                const float2 ml = region(w)[kMaxNt * 32 + lane];
                sc[w] = exp2_diff(ml.x, M);
                Lsum += sc[w] * ml.y;
            }
        }
    };
    auto merged_pair = [&](const float (&sc)[kMmaWarps], int x) -> float2 {
        float2 v = make_float2(0.f, 0.f);
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w)
            if (sc[w] != 0.f) {
                const float2 t = region(w)[x * 32 + lane];
                v.x += sc[w] * t.x;
                v.y += sc[w] * t.y;
            }
        return v;
    };

    for (;;) {
        if (!warp_wait(bar(B_MF), ndump & 1, p.status)) return false;
        const int kind = dsc[0];
        if (kind == kDumpEnd) return true;
        const int g = dsc[1], rv8 = dsc[2], flags = dsc[3], recslot = dsc[4], pass = dsc[5];
        const int item = dsc[6], qi = dsc[7];
        if (kind == kDumpSeg) {
            const int pb = npv & 1;
            if (!warp_wait(bar(B_PVF0 + pb), (npv / 2) & 1, p.status)) return false;
            const uint32_t pv = pv_base + pb * L::kPBytes;
            const int nkj = (rv8 + 15) / 16, nvt = rv8 / 8;
            const int ngrp = p.nrg_cta;
            // the dump regions are free once the last row group is merged
            int last_grp = 0;
            for (int x = 0; x < ngrp; ++x)
                if (pass * ngrp + x < p.nrg) last_grp = x;
            bool me_done = false;
#pragma unroll
            for (int grp = 0; grp < 2; ++grp) {
                if (grp >= ngrp) break;
                const int rg = pass * ngrp + grp;
                if (rg >= p.nrg) continue;
                float sc[kMmaWarps], M, Lsum;
                merge_scales(ngrp, grp, sc, M, Lsum);
                if (flags & F_RUN_FIRST) {
                    m_run[grp] = -INFINITY;
                    l_run[grp] = 0.f;
#pragma unroll
                    for (int x = 0; x < kHalf; ++x) orun[grp][x][0] = orun[grp][x][1] = 0.f;
                }
                const float m_new = fmaxf(m_run[grp], M);
                const float a_run = exp2_diff(m_run[grp], m_new), a_seg = exp2_diff(M, m_new);
#pragma unroll
                for (int w = 0; w < kMmaWarps; ++w) sc[w] *= a_seg;
                uint32_t af[kMaxKs][4];
#pragma unroll
                for (int kj = 0; kj < kMaxKs; ++kj) {
                    if (kj < nkj) {
                        const float2 x = (2 * kj < nvt) ? merged_pair(sc, 2 * kj) : make_float2(0.f, 0.f);
                        const float2 y = (2 * kj + 1 < nvt) ? merged_pair(sc, 2 * kj + 1) : make_float2(0.f, 0.f);
                        split_hi_lo(x.x, x.y, af[kj][0], af[kj][1]);
                        split_hi_lo(y.x, y.y, af[kj][2], af[kj][3]);
                    }
                }
                if (grp == last_grp) {
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar(B_ME));
                    me_done = true;
                }
                // back-projection through P^V into this warp's half of the run's output
                const int mi = lane / 8;
#pragma unroll
                for (int cp = 0; cp < kHalf / 2; ++cp) {
                    float oa[4] = {0.f, 0.f, 0.f, 0.f}, ob[4] = {0.f, 0.f, 0.f, 0.f};
                    // tiles (2kj, c), (2kj+1, c), (2kj, c+1), (2kj+1, c+1) of P^V, c = ct0 + 2cp
                    const int ct = ct0 + 2 * cp + (mi >> 1);
#pragma unroll
                    for (int kj = 0; kj < kMaxKs; ++kj) {
                        if (kj < nkj) {
                            const int jg = 2 * kj + (mi & 1);
                            const uint32_t addr =
                                (jg < rv8 / 8) ? pv + (jg * (D / 8) + ct) * 128 + (lane % 8) * 16 : zero_addr;
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4_t(addr, b0, b1, b2, b3);
                            mma16816(oa, af[kj], b0, b1);
                            mma16816(ob, af[kj], b2, b3);
                        }
                    }
                    orun[grp][2 * cp][0] = orun[grp][2 * cp][0] * a_run + (oa[0] + oa[2]);
                    orun[grp][2 * cp][1] = orun[grp][2 * cp][1] * a_run + (oa[1] + oa[3]);
                    orun[grp][2 * cp + 1][0] = orun[grp][2 * cp + 1][0] * a_run + (ob[0] + ob[2]);
                    orun[grp][2 * cp + 1][1] = orun[grp][2 * cp + 1][1] * a_run + (ob[1] + ob[3]);
                }
                l_run[grp] = l_run[grp] * a_run + Lsum * a_seg;
                m_run[grp] = m_new;
            }
            __syncwarp();
            if (lane == 0) {
                if (!me_done) mbar_arrive(bar(B_ME));
                mbar_arrive(bar(B_PVE0 + pb));
            }
            ++npv;
            if (flags & F_RUN_LAST) {
#pragma unroll
                for (int grp = 0; grp < 2; ++grp) {
                    if (grp >= ngrp) break;
                    const int rg = pass * ngrp + grp;
                    if (rg >= p.nrg) continue;
                    float *rec = p.rec + ((int64_t)recslot * p.nrg + rg) * recf;
#pragma unroll
                    for (int x = 0; x < kHalf; ++x)
                        __stcg(reinterpret_cast<float2 *>(rec + quad * D + 8 * (ct0 + x) + 2 * qlane),
                               make_float2(orun[grp][x][0], orun[grp][x][1]));
                    if (ep == 0 && qlane == 0) {
                        __stcg(rec + 8 * D + quad, m_run[grp]);
                        __stcg(rec + 8 * D + 8 + quad, l_run[grp]);
                    }
                    __threadfence();
                    if (!await_partner()) return false;
                    if (ep == 0) ticket(g, rg);
                }
            }
        } else {  // tail item: the merged accumulator is already the output
            const int ngrp = p.ngrp_t;
            for (int grp = 0; grp < ngrp; ++grp) {
                const int rgt = pass * ngrp + grp;
                if (rgt >= p.nrg_t) continue;
                float sc[kMmaWarps], M, Lsum;
                merge_scales(ngrp, grp, sc, M, Lsum);
                float *rec = p.rec + (p.tail_rec_base + (int64_t)item * p.nrg_t + rgt) * recf;
#pragma unroll
                for (int x = 0; x < kHalf; ++x)
                    __stcg(reinterpret_cast<float2 *>(rec + quad * D + 8 * (ct0 + x) + 2 * qlane),
                           merged_pair(sc, ct0 + x));
                if (ep == 0 && qlane == 0) {
                    __stcg(rec + 8 * D + quad, M);
                    __stcg(rec + 8 * D + 8 + quad, Lsum);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(B_ME));
            __threadfence();
            if (!await_partner()) return false;
            if (ep == 1) {
                ++ndump;
                continue;
            }
            // tickets of the prefix row groups these query rows belong to
            for (int grp = 0; grp < ngrp; ++grp) {
                const int rgt = pass * ngrp + grp;
                if (rgt >= p.nrg_t) continue;
                const int ra = qi * p.G + 8 * rgt, rb = qi * p.G + min(8 * rgt + 8, p.G);  // [ra, rb)
                for (int rg = ra / 8; rg <= (rb - 1) / 8; ++rg) ticket(g, rg);
            }
        }
        ++ndump;
    }
}

// ================================================================ kernel
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    decode_kernel(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_v)
{
    using L = Lay<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    int32_t *hdr = reinterpret_cast<int32_t *>(smem + L::kHdr);
    int32_t *pkh = hdr + kSlots * kHdrInts;
    int32_t *dsc = hdr + (kSlots + 1) * kHdrInts;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L::kBar);
    int32_t *list = reinterpret_cast<int32_t *>(smem + L::kList);
    const uint32_t zero_addr = smem_u32(smem + L::kZero);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

    pdl_trigger();
    if (threadIdx.x == 0) {
        for (int s = 0; s < kSlots; ++s) {
            mbar_init(smem_u32(&bars[s]), 1);                    // full: producer + bytes
            mbar_init(smem_u32(&bars[kSlots + s]), kMmaWarps);   // empty: every MMA warp
        }
        mbar_init(smem_u32(&bars[B_PKF]), 1);
        mbar_init(smem_u32(&bars[B_PKE]), 1);
        mbar_init(smem_u32(&bars[B_PVF0]), 1);
        mbar_init(smem_u32(&bars[B_PVF1]), 1);
        mbar_init(smem_u32(&bars[B_PVE0]), 2);  // both epilogue warps
        mbar_init(smem_u32(&bars[B_PVE1]), 2);
        mbar_init(smem_u32(&bars[B_QR]), 1);
        mbar_init(smem_u32(&bars[B_QF]), kMmaWarps);
        mbar_init(smem_u32(&bars[B_MF]), kMmaWarps);
        mbar_init(smem_u32(&bars[B_ME]), 2);   // both epilogue warps
        mbar_init(smem_u32(&bars[B_EPS]), 2);
        mbar_init(smem_u32(&bars[B_FIN]), 3 + kMmaWarps);
        list[0] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x < 32) reinterpret_cast<uint32_t *>(smem + L::kZero)[threadIdx.x] = 0u;
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) run_producer<D>(p, smem, hdr, pkh, bars, &tmap_k, &tmap_v);
        return;
    }
    bool ok;
    if (warp == 1)
        ok = run_projection<D>(p, smem, pkh, bars, lane);
    else if (warp <= 3)
        ok = run_epilogue<D>(p, smem, dsc, bars, list, zero_addr, warp - 2, lane);
    else
        ok = run_mma<D>(p, smem, hdr, dsc, bars, zero_addr, warp - 4, lane);
    if (!ok) return;
    // every role done: merge the row groups this thread block completed
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&bars[B_FIN]));
    if (!warp_wait(smem_u32(&bars[B_FIN]), 0, p.status)) return;
    const int n = min(list[0], L::kListCap);
    for (int k = 0; k < n; ++k)
        combine_rows<D>(p, list[1 + 2 * k], list[2 + 2 * k], threadIdx.x - 32, kThreads - 32);
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
    constexpr int kMaxDevices = 64;
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
    static int configured[2] = {0, 0};  // largest dynamic smem size set per kernel
    const int which = p.d == 64 ? 0 : 1;
    if (smem_bytes > configured[which]) {
        cudaError_t e = which == 0 ? cudaFuncSetAttribute(decode_kernel<64>,
                                                          cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes)
                                   : cudaFuncSetAttribute(decode_kernel<128>,
                                                          cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
        if (e != cudaSuccess) return e;
        configured[which] = smem_bytes;
    }
    if (which == 0) return cudaLaunchKernelEx(&cfg, decode_kernel<64>, p, mk, mv);
    return cudaLaunchKernelEx(&cfg, decode_kernel<128>, p, mk, mv);
}

}  // namespace milo
