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
// One persistent thread block per SM.  Warp 0 is the producer: one lane walks
// the block's static list of prefix segments (and afterwards grabs dense-tail
// items from a counter), writes a small header into the next ring slot and
// starts a 1-D bulk copy (packed factors) or a 3-D tensor copy (tail) into
// it, completing on the slot's mbarrier.  Warps 1..8 are consumers: they
// follow the headers.  A segment is
//     [P^K]  -> q~ = scale*log2(e) * P^K q for the segment's query rows
//     [C^K C^V]... -> 16-token sub-tiles round-robin over the warps:
//                   scores (mma m16n8k16, q~ split into bf16 hi+lo in the
//                   16 A rows), online softmax in registers, rank-space value
//                   accumulation (p split into bf16 hi+lo in the A rows)
//     [P^V]  -> merge the warps' (max, sum, v~), back-project v~ P^V into the
//               head dimension and fold into the run's running output.
// The last segment of a run (same KV head, same thread block) writes a
// partial record (o[8][d], m[8], l[8]); the last record of a (KV head, row
// group) to arrive -- counted with a ticket, no waiting -- merges all records
// of those rows and writes the fp32 output.
//
// Every mbarrier wait is bounded (about 2 s of wall time); on expiry the
// thread records MILO_ERR_TIMEOUT in the sticky status word and leaves.
#include <cuda.h>
#include <cuda_bf16.h>

#include "milo.h"
#include "milo_internal.h"

namespace milo {
namespace {

constexpr uint64_t kTimeoutNs = 2000000000ull;

enum : int { kEnd = 0, kPK = 1, kC = 2, kPV = 3, kTail = 4 };

// header words
enum : int {
    H_KIND = 0, H_E = 1, H_G = 2, H_T0 = 3, H_T1 = 4, H_RK8 = 5, H_RV8 = 6,
    H_PASS = 7, H_FLAGS = 8, H_REC = 9, H_QI = 10, H_TOK8 = 11, H_NSUB = 12
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
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(tx)
                 : "memory");
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

// Barrier among the warps of one group, built on an mbarrier whose arrival
// count is the group's warp count, so that it waits with the same time limit
// as every other wait.  `phases` holds one phase bit per barrier index.
__device__ __forceinline__ bool group_sync(uint64_t *bar, uint32_t &phases, int idx, int lane, int32_t *status)
{
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(bar));
    const bool ok = warp_wait(smem_u32(bar), (phases >> idx) & 1u, status);
    phases ^= 1u << idx;
    return ok;
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
struct SmemLayout {
    static constexpr int kKSteps = D / 16;               // max q~ k-steps (r8 <= D)
    static constexpr int kQsBytes = kKSteps * 32 * 16;   // per parity
    static constexpr int kVaBytes = 8 * D * 4;           // per parity
    static constexpr int kMlBytes = kConsumerWarps * 8 * 2 * 4;  // per parity
    static constexpr int kGroupBytes = 2 * (kQsBytes + kVaBytes + kMlBytes);
    static constexpr int kHdrOff = kSlots * kSlotBytes;
    static constexpr int kBarOff = kHdrOff + kSlots * kHdrInts * 4;
    static constexpr int kGBars = 9;  // 4 prefix groups, 4 tail groups, all consumers
    static constexpr int kZeroOff = kBarOff + (2 * kSlots + kGBars) * 8;
    static constexpr int kFlagOff = kZeroOff + 128;      // per-group broadcast ints
    static constexpr int kGroupOff = kFlagOff + 128;
    static int bytes(int groups) { return kGroupOff + groups * kGroupBytes + 1024; }
};

template <int D>
struct Group {
    uint4 *qs[2];
    float *va[2];
    float *ml[2];
};

template <int D>
__device__ __forceinline__ Group<D> group_ptrs(uint8_t *base, int grp)
{
    using L = SmemLayout<D>;
    uint8_t *g = base + L::kGroupOff + grp * L::kGroupBytes;
    Group<D> r;
    r.qs[0] = reinterpret_cast<uint4 *>(g);
    r.qs[1] = reinterpret_cast<uint4 *>(g + L::kQsBytes);
    r.va[0] = reinterpret_cast<float *>(g + 2 * L::kQsBytes);
    r.va[1] = reinterpret_cast<float *>(g + 2 * L::kQsBytes + L::kVaBytes);
    r.ml[0] = reinterpret_cast<float *>(g + 2 * L::kQsBytes + 2 * L::kVaBytes);
    r.ml[1] = reinterpret_cast<float *>(g + 2 * L::kQsBytes + 2 * L::kVaBytes + L::kMlBytes);
    return r;
}

// ------------------------------------------------------- combine ----------
// Merge every partial record of (KV head g, row group rg) and write out.
// Executed by `nthr` threads (tid in [0, nthr)) of one warp group.
template <int D>
__device__ void combine_rows(const DecodeParams &p, int g, int rg, int tid, int nthr)
{
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
        auto rec_of = [&](int s, int &row) -> const float * {
            if (s < nprefix) {
                row = k;
                return p.rec + (int64_t)((gs0 + s) * p.nrg + rg) * recf;
            }
            const int t = s - nprefix;
            row = hh % 8;
            return p.rec + (p.tail_rec_base + ((int64_t)(i * p.hkv + g) * S + t) * p.nrg_t + hh / 8) * recf;
        };
        float M = -INFINITY;
#pragma unroll 8
        for (int s = 0; s < nsrc; ++s) {
            int row;
            const float *r = rec_of(s, row);
            M = fmaxf(M, __ldcg(r + 8 * D + row));
        }
        float L = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
        for (int s = 0; s < nsrc; ++s) {
            int row;
            const float *r = rec_of(s, row);
            const float m = __ldcg(r + 8 * D + row);
            const float l = __ldcg(r + 8 * D + 8 + row);
            const float4 o = __ldcg(reinterpret_cast<const float4 *>(r + row * D) + c4);
            const float w8 = exp2_diff(m, M);
            L += w8 * l;
            acc.x += w8 * o.x;
            acc.y += w8 * o.y;
            acc.z += w8 * o.z;
            acc.w += w8 * o.w;
        }
        const float inv = 1.f / L;
        float4 res = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
        float *dst = p.out + ((int64_t)i * p.hq + g * p.G + hh) * D;
        reinterpret_cast<float4 *>(dst)[c4] = res;
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

// ------------------------------------------------------- the kernel -------
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    decode_kernel(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_v)
{
    using L = SmemLayout<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    int32_t *hdr_all = reinterpret_cast<int32_t *>(smem + L::kHdrOff);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L::kBarOff);
    int32_t *flags = reinterpret_cast<int32_t *>(smem + L::kFlagOff);
    const uint32_t zero_addr = smem_u32(smem + L::kZeroOff);
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int ngroups_alloc = max(p.nrg_cta, p.nrg_t <= 1 ? 1 : (p.nrg_t <= 2 ? 2 : 4));

    pdl_trigger();

    if (threadIdx.x == 0) {
        for (int s = 0; s < kSlots; ++s) {
            mbar_init(smem_u32(&bars[s]), 1);                        // full
            mbar_init(smem_u32(&bars[kSlots + s]), kConsumerWarps);  // empty
        }
        const int ngrp_t = p.nrg_t <= 1 ? 1 : (p.nrg_t <= 2 ? 2 : 4);
        for (int x = 0; x < 4; ++x) {
            mbar_init(smem_u32(&bars[2 * kSlots + x]), kConsumerWarps / p.nrg_cta);  // prefix groups
            mbar_init(smem_u32(&bars[2 * kSlots + 4 + x]), kConsumerWarps / ngrp_t);  // tail groups
        }
        mbar_init(smem_u32(&bars[2 * kSlots + 8]), kConsumerWarps);                 // all consumers
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x < 32) reinterpret_cast<uint32_t *>(smem + L::kZeroOff)[threadIdx.x] = 0u;
    // zero the merge accumulators of every group, both parities
    for (int grp = 0; grp < ngroups_alloc; ++grp) {
        Group<D> G = group_ptrs<D>(smem, grp);
        for (int x = threadIdx.x; x < 2 * 8 * D; x += blockDim.x) (x < 8 * D ? G.va[0] : G.va[1])[x % (8 * D)] = 0.f;
    }
    __syncthreads();

    const int cta = blockIdx.x;

    // ================================================================ producer
    if (warp == 0) {
        if (lane != 0) return;
        int seq = 0;
        auto acquire = [&](int kind) -> int {
            const int slot = seq % kSlots;
            if (seq >= kSlots) {
                if (!mbar_wait(smem_u32(&bars[kSlots + slot]), ((seq / kSlots) - 1) & 1, p.status)) return -1;
            }
            int32_t *h = hdr_all + slot * kHdrInts;
            h[H_KIND] = kind;
            return slot;
        };
        auto commit = [&](int slot, uint32_t bytes) {
            (void)bytes;
            ++seq;
        };
        bool ok = true;
        const int s_begin = p.cta_seg_begin[cta], s_end = p.cta_seg_begin[cta + 1];
        for (int s = s_begin; s < s_end && ok;) {
            int r1 = s;
            while (r1 < s_end - 1 && !(p.segs[r1].flags & kSegLastOfRun)) ++r1;
            for (int pass = 0; pass < p.npass && ok; ++pass) {
                for (int sg = s; sg <= r1 && ok; ++sg) {
                    const SegDev seg = p.segs[sg];
                    const EntryDev ent = p.entries[seg.entry];
                    const int rk8 = (ent.rk + 7) & ~7, rv8 = (ent.rv + 7) & ~7;
                    int fl = 0;
                    if (sg == s) fl |= kSegFirstOfRun;
                    if (sg == r1) fl |= kSegLastOfRun;
                    // --- P^K
                    int slot = acquire(kPK);
                    if (slot < 0) { ok = false; break; }
                    {
                        int32_t *h = hdr_all + slot * kHdrInts;
                        h[H_E] = seg.entry; h[H_G] = ent.g; h[H_T0] = seg.t0; h[H_T1] = seg.t1;
                        h[H_RK8] = rk8; h[H_RV8] = rv8; h[H_PASS] = pass; h[H_FLAGS] = fl; h[H_REC] = seg.slot;
                        const uint32_t bar = smem_u32(&bars[slot]);
                        const uint32_t bytes = (uint32_t)rk8 * D * 2;
                        if (bytes) {
                            mbar_arrive_tx(bar, bytes);
                            bulk_g2s(smem_u32(smem + slot * kSlotBytes), p.packed + ent.off_pk, bytes, bar);
                        } else {
                            mbar_arrive(bar);
                        }
                        commit(slot, bytes);
                    }
                    // --- coefficient tiles
                    const int per_tile = kTileTokens * (rk8 + rv8) * 2;
                    int tiles_per_slot = per_tile > 0 ? kSlotBytes / per_tile : 8;
                    tiles_per_slot = max(1, min(tiles_per_slot, 8));
                    const int n8 = (ent.n + 7) & ~7;
                    for (int tt0 = seg.t0; tt0 < seg.t1 && ok; tt0 += tiles_per_slot * kTileTokens) {
                        const int tt1 = min(seg.t1, tt0 + tiles_per_slot * kTileTokens);
                        const int tok8 = min(((tt1 + 7) & ~7), n8) - tt0;
                        const int ntl = (tt1 - tt0 + kTileTokens - 1) / kTileTokens;
                        const int last8 = tok8 - (ntl - 1) * kTileTokens;
                        const int nsub = 4 * (ntl - 1) + (last8 + 15) / 16;
                        slot = acquire(kC);
                        if (slot < 0) { ok = false; break; }
                        int32_t *h = hdr_all + slot * kHdrInts;
                        h[H_E] = seg.entry; h[H_G] = ent.g; h[H_T0] = tt0; h[H_T1] = tt1;
                        h[H_RK8] = rk8; h[H_RV8] = rv8; h[H_PASS] = pass; h[H_FLAGS] = fl;
                        h[H_REC] = seg.slot; h[H_TOK8] = tok8; h[H_NSUB] = nsub;
                        const uint32_t kb = (uint32_t)tok8 * rk8 * 2, vb = (uint32_t)tok8 * rv8 * 2;
                        const uint32_t bar = smem_u32(&bars[slot]);
                        if (kb + vb) {
                            mbar_arrive_tx(bar, kb + vb);
                            const uint32_t dst = smem_u32(smem + slot * kSlotBytes);
                            if (kb) bulk_g2s(dst, p.packed + ent.off_ck + (int64_t)tt0 * rk8 * 2, kb, bar);
                            if (vb) bulk_g2s(dst + kb, p.packed + ent.off_cv + (int64_t)tt0 * rv8 * 2, vb, bar);
                        } else {
                            mbar_arrive(bar);
                        }
                        commit(slot, kb + vb);
                    }
                    if (!ok) break;
                    // --- P^V
                    slot = acquire(kPV);
                    if (slot < 0) { ok = false; break; }
                    {
                        int32_t *h = hdr_all + slot * kHdrInts;
                        h[H_E] = seg.entry; h[H_G] = ent.g; h[H_T0] = seg.t0; h[H_T1] = seg.t1;
                        h[H_RK8] = rk8; h[H_RV8] = rv8; h[H_PASS] = pass; h[H_FLAGS] = fl; h[H_REC] = seg.slot;
                        const uint32_t bar = smem_u32(&bars[slot]);
                        const uint32_t bytes = (uint32_t)rv8 * D * 2;
                        if (bytes) {
                            mbar_arrive_tx(bar, bytes);
                            bulk_g2s(smem_u32(smem + slot * kSlotBytes), p.packed + ent.off_pv, bytes, bar);
                        } else {
                            mbar_arrive(bar);
                        }
                        commit(slot, bytes);
                    }
                }
            }
            s = r1 + 1;
        }
        // Dense tails: read after the preceding grid has completed.
        pdl_wait();
        if (ok && p.has_tail) {
            const int S = p.tail_splits;
            for (;;) {
                const uint32_t item = atomicAdd(&p.counters->tail_next, 1u);
                if (item >= (uint32_t)p.num_tail_items) break;
                const int i = item / (p.hkv * S), g = (item / S) % p.hkv, sp = item % S;
                const int64_t o0 = p.tail_offsets[i], o1 = p.tail_offsets[i + 1];
                const int T = (int)(o1 - o0);
                if (sp == S - 1 && T > S * kTailTokens) atomicCAS(p.status, 0, (int32_t)MILO_ERR_DEVICE_BOUNDS);
                const int t0 = sp * kTailTokens, t1 = min(t0 + kTailTokens, T);
                const int slot = acquire(kTail);
                if (slot < 0) { ok = false; break; }
                int32_t *h = hdr_all + slot * kHdrInts;
                h[H_E] = (int)item; h[H_G] = g; h[H_QI] = i; h[H_T0] = t0; h[H_T1] = t1;
                const uint32_t bar = smem_u32(&bars[slot]);
                if (t1 > t0) {
                    constexpr uint32_t half = 64 * 64 * 2;  // one 64-token x 64-column box
                    constexpr uint32_t bytes = 2 * (D / 64) * half;
                    mbar_arrive_tx(bar, bytes);
                    const uint32_t dst = smem_u32(smem + slot * kSlotBytes);
                    const int row = (int)(o0 + t0);
#pragma unroll
                    for (int hb = 0; hb < D / 64; ++hb) {
                        tma_load_3d(dst + hb * half, &tmap_k, 64 * hb, g, row, bar);
                        tma_load_3d(dst + (D / 64) * half + hb * half, &tmap_v, 64 * hb, g, row, bar);
                    }
                } else {
                    mbar_arrive(bar);
                }
                commit(slot, 0);
            }
        }
        if (ok) {
            const int slot = acquire(kEnd);
            if (slot >= 0) {
                mbar_arrive(smem_u32(&bars[slot]));
                commit(slot, 0);
            }
        }
        // the last thread block to finish grabbing resets the tail counter
        if (atomicAdd(&p.counters->ctas_done, 1u) == (uint32_t)p.num_ctas - 1) {
            p.counters->tail_next = 0u;
            p.counters->ctas_done = 0u;
        }
        // do not leave while a copy this thread started may still be landing
        for (int j = max(0, seq - kSlots); j < seq; ++j)
            if (!mbar_wait(smem_u32(&bars[j % kSlots]), (j / kSlots) & 1, p.status)) break;
        return;
    }

    // ================================================================ consumers
    const int cw = warp - 1;
    const int quad = lane / 4, qlane = lane % 4;
    constexpr int kMaxNt = D / 8;   // max rank (or column) 8-tiles
    constexpr int kMaxKs = D / 16;  // max 16-wide k-steps

    pdl_wait();  // q, tails and the workspace belong to the preceding grid until here

    uint32_t qf[kMaxKs][4];
    float vacc[kMaxNt][4];
    float orun[kMaxNt / 2][2];  // own back-projection column tiles (TS >= 2)
    float m_w = -INFINITY, l_w = 0.f;
    float m_run = -INFINITY, l_run = 0.f;
    int par[4] = {0, 0, 0, 0};
    int sub_base = 0;
    bool tail_phase = false;
    uint32_t gph = 0;  // phase bits of the group barriers

#pragma unroll
    for (int x = 0; x < kMaxNt / 2; ++x) orun[x][0] = orun[x][1] = 0.f;

    for (int seq = 0;; ++seq) {
        const int slot = seq % kSlots;
        if (!warp_wait(smem_u32(&bars[slot]), (seq / kSlots) & 1, p.status)) return;
        const int32_t *h = hdr_all + slot * kHdrInts;
        const int kind = h[H_KIND];
        if (kind == kEnd) break;
        const uint32_t sbase = smem_u32(smem + slot * kSlotBytes);

        if (kind == kTail && !tail_phase) {
            // switch every warp to the tail grouping with fresh merge buffers
            if (!group_sync(&bars[2 * kSlots + 8], gph, 8, lane, p.status)) return;
            for (int grp = 0; grp < ngroups_alloc; ++grp) {
                Group<D> Gp = group_ptrs<D>(smem, grp);
                for (int x = cw * 32 + lane; x < 2 * 8 * D; x += kConsumerWarps * 32)
                    (x < 8 * D ? Gp.va[0] : Gp.va[1])[x % (8 * D)] = 0.f;
            }
            if (!group_sync(&bars[2 * kSlots + 8], gph, 8, lane, p.status)) return;
            par[0] = par[1] = par[2] = par[3] = 0;
            sub_base = 0;
            tail_phase = true;
        }

        // --- warp group of this header
        int ngrp, grp_sz;
        if (kind == kTail) {
            ngrp = p.nrg_t <= 1 ? 1 : (p.nrg_t <= 2 ? 2 : 4);
        } else {
            ngrp = p.nrg_cta;
        }
        grp_sz = kConsumerWarps / ngrp;              // warps per group (TS)
        const int grp = cw % ngrp, phase = cw / ngrp;
        const int bidx = (kind == kTail ? 4 : 0) + grp, bar_n = grp_sz * 32;
        uint64_t *gbar = &bars[2 * kSlots + bidx];
        Group<D> GB = group_ptrs<D>(smem, grp);
        const int g = h[H_G];

        if (kind == kPK || kind == kC || kind == kPV) {
            const int rg = h[H_PASS] * p.nrg_cta + grp;
            const bool active = rg < p.nrg;
            const int rk8 = h[H_RK8], rv8 = h[H_RV8];
            if (active && kind == kPK) {
                const int pp = par[grp];
                // q rows of this row group (bf16, exact) as A fragments; lo rows zero
                const int rho = 8 * rg + quad;
                const uint16_t *qrow = nullptr;
                if (rho < p.rows_g) {
                    const int i = rho / p.G, hh = rho % p.G;
                    qrow = p.q + ((int64_t)i * p.hq + g * p.G + hh) * D;
                }
                uint32_t qlo[kMaxKs], qhi[kMaxKs];
#pragma unroll
                for (int kc = 0; kc < kMaxKs; ++kc) {
                    qlo[kc] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 2 * qlane) : 0u;
                    qhi[kc] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 8 + 2 * qlane) : 0u;
                }
                const int njt = 2 * ((rk8 + 15) / 16);
                for (int jt = phase; jt < njt; jt += grp_sz) {
                    float acc[4] = {0.f, 0.f, 0.f, 0.f};
                    if (jt < rk8 / 8) {
#pragma unroll
                        for (int kc = 0; kc < kMaxKs; kc += 2) {
                            uint32_t b0, b1, b2, b3;
                            // tiles (jt, 2kc), (jt, 2kc+1), (jt, 2kc+2), (jt, 2kc+3) of P^K
                            const int cg = 2 * kc + (lane / 8);
                            ldsm_x4(sbase + (jt * (D / 8) + cg) * 128 + (lane % 8) * 16, b0, b1, b2, b3);
                            const uint32_t a0[4] = {qlo[kc], 0u, qhi[kc], 0u};
                            const uint32_t a1[4] = {qlo[kc + 1], 0u, qhi[kc + 1], 0u};
                            mma16816(acc, a0, b0, b1);
                            mma16816(acc, a1, b2, b3);
                        }
                    }
                    uint32_t hi, lo;
                    split_hi_lo(acc[0] * p.scale_log2, acc[1] * p.scale_log2, hi, lo);
                    uint32_t *dst = reinterpret_cast<uint32_t *>(GB.qs[pp] + (jt / 2) * 32 + lane);
                    dst[(jt & 1) * 2 + 0] = hi;
                    dst[(jt & 1) * 2 + 1] = lo;
                }
                if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                const int nks = (rk8 + 15) / 16;
#pragma unroll
                for (int kk = 0; kk < kMaxKs; ++kk) {
                    if (kk < nks) {
                        const uint4 v = GB.qs[pp][kk * 32 + lane];
                        qf[kk][0] = v.x; qf[kk][1] = v.y; qf[kk][2] = v.z; qf[kk][3] = v.w;
                    }
                }
                m_w = -INFINITY;
                l_w = 0.f;
#pragma unroll
                for (int x = 0; x < kMaxNt; ++x) vacc[x][0] = vacc[x][1] = vacc[x][2] = vacc[x][3] = 0.f;
                if (h[H_FLAGS] & kSegFirstOfRun) {
                    m_run = -INFINITY;
                    l_run = 0.f;
#pragma unroll
                    for (int x = 0; x < kMaxNt / 2; ++x) orun[x][0] = orun[x][1] = 0.f;
                }
            } else if (active && kind == kC) {
                const int t0 = h[H_T0], t1 = h[H_T1], tok8 = h[H_TOK8], nsub = h[H_NSUB];
                const uint32_t kbase = sbase, vbase = sbase + tok8 * rk8 * 2;
                const int nks = (rk8 + 15) / 16, njp = (rv8 + 15) / 16;
                const int ntl = (t1 - t0 + kTileTokens - 1) / kTileTokens;
                for (int u = 0; u < nsub; ++u) {
                    if ((sub_base + u) % grp_sz != phase) continue;
                    const int kt = u / 4, su = u % 4;
                    const int t8 = (kt == ntl - 1) ? tok8 - kt * kTileTokens : kTileTokens;
                    const int ntg = t8 / 8;
                    const int tga = 2 * su, tgb = tga + 1;
                    const uint32_t ktile = kbase + kt * kTileTokens * rk8 * 2;
                    const uint32_t vtile = vbase + kt * kTileTokens * rv8 * 2;
                    float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
                    {
                        const int mi = lane / 8;
                        const int tg = (mi < 2) ? tga : tgb;
#pragma unroll
                        for (int kk = 0; kk < kMaxKs; ++kk) {
                            if (kk < nks) {
                                const int rgk = 2 * kk + (mi & 1);
                                const uint32_t addr = (tg < ntg && rgk < rk8 / 8)
                                                          ? ktile + (rgk * ntg + tg) * 128 + (lane % 8) * 16
                                                          : zero_addr;
                                uint32_t b0, b1, b2, b3;
                                ldsm_x4(addr, b0, b1, b2, b3);
                                mma16816(sa, qf[kk], b0, b1);
                                mma16816(sb, qf[kk], b2, b3);
                            }
                        }
                    }
                    const int tokA = t0 + kt * kTileTokens + 8 * tga + 2 * qlane;
                    const int tokB = tokA + 8;
                    float s0 = sa[0] + sa[2], s1 = sa[1] + sa[3], s2 = sb[0] + sb[2], s3 = sb[1] + sb[3];
                    if (tokA >= t1) s0 = -INFINITY;
                    if (tokA + 1 >= t1) s1 = -INFINITY;
                    if (tokB >= t1 || tgb >= ntg) s2 = -INFINITY;
                    if (tokB + 1 >= t1 || tgb >= ntg) s3 = -INFINITY;
                    const float mx = quad_max(fmaxf(fmaxf(s0, s1), fmaxf(s2, s3)));
                    if (mx > m_w + 8.f) {
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
                    {
                        const int mi = lane / 8;
                        const int tg = (mi & 1) ? tgb : tga;
#pragma unroll
                        for (int jp = 0; jp < kMaxKs; ++jp) {
                            if (jp < njp) {
                                const int rgv = 2 * jp + (mi >> 1);
                                const uint32_t addr = (tg < ntg && rgv < rv8 / 8)
                                                          ? vtile + (rgv * ntg + tg) * 128 + (lane % 8) * 16
                                                          : zero_addr;
                                uint32_t b0, b1, b2, b3;
                                ldsm_x4_t(addr, b0, b1, b2, b3);
                                mma16816(vacc[2 * jp], pa, b0, b1);
                                mma16816(vacc[2 * jp + 1], pa, b2, b3);
                            }
                        }
                    }
                }
                sub_base += nsub;
            } else if (active && kind == kPV) {
                const int pp = par[grp];
                // 1-2: publish this warp's running max and sum
                const float lq = quad_sum(l_w);
                if (qlane == 0) {
                    GB.ml[pp][(phase * 8 + quad) * 2 + 0] = m_w;
                    GB.ml[pp][(phase * 8 + quad) * 2 + 1] = lq;
                }
                if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                // 3: merged max / sum of the segment; scale own v~ into the shared sum
                float m_seg = -INFINITY;
                for (int w = 0; w < grp_sz; ++w) m_seg = fmaxf(m_seg, GB.ml[pp][(w * 8 + quad) * 2]);
                float l_seg = 0.f;
                for (int w = 0; w < grp_sz; ++w)
                    l_seg += exp2_diff(GB.ml[pp][(w * 8 + quad) * 2], m_seg) * GB.ml[pp][(w * 8 + quad) * 2 + 1];
                const float sc = exp2_diff(m_w, m_seg);
                const int nvt = rv8 / 8;
                float *va = GB.va[pp];
#pragma unroll
                for (int x = 0; x < kMaxNt; ++x) {
                    if (x < nvt && sc != 0.f) {
                        const int j = 8 * x + 2 * qlane;
                        atomicAdd(&va[quad * D + j], (vacc[x][0] + vacc[x][2]) * sc);
                        atomicAdd(&va[quad * D + j + 1], (vacc[x][1] + vacc[x][3]) * sc);
                    }
                }
                if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                // 4: back-projection o = v~ P^V for this warp's column tiles, folded
                //    straight into the run's output (scaled to the new running max)
                const int nkj = (rv8 + 15) / 16;
                const float m_new = fmaxf(m_run, m_seg);
                const float a_run = exp2_diff(m_run, m_new), a_seg = exp2_diff(m_seg, m_new);
#pragma unroll
                for (int x = 0; x < kMaxNt / 2; ++x) { orun[x][0] *= a_run; orun[x][1] *= a_run; }
#pragma unroll
                for (int xp = 0; xp < kMaxNt / 4; ++xp) {
                    const int cta_ = phase + (2 * xp) * grp_sz, ctb = phase + (2 * xp + 1) * grp_sz;
                    if (cta_ < kMaxNt) {
                        float oa[4] = {0.f, 0.f, 0.f, 0.f}, ob[4] = {0.f, 0.f, 0.f, 0.f};
                        const int mi = lane / 8;  // tiles (2kj, cta), (2kj+1, cta), (2kj, ctb), (2kj+1, ctb)
                        const int ct = (mi < 2) ? cta_ : ctb;
#pragma unroll
                        for (int kj = 0; kj < kMaxKs; ++kj) {
                            if (kj < nkj) {
                                const float2 x = *reinterpret_cast<const float2 *>(&va[quad * D + 16 * kj + 2 * qlane]);
                                const float2 y = *reinterpret_cast<const float2 *>(&va[quad * D + 16 * kj + 8 + 2 * qlane]);
                                uint32_t af[4];
                                split_hi_lo(x.x * a_seg, x.y * a_seg, af[0], af[1]);
                                split_hi_lo(y.x * a_seg, y.y * a_seg, af[2], af[3]);
                                const int jg = 2 * kj + (mi & 1);
                                const uint32_t addr = (jg < rv8 / 8 && ct < kMaxNt)
                                                          ? sbase + (jg * (D / 8) + ct) * 128 + (lane % 8) * 16
                                                          : zero_addr;
                                uint32_t b0, b1, b2, b3;
                                ldsm_x4_t(addr, b0, b1, b2, b3);
                                mma16816(oa, af, b0, b1);
                                mma16816(ob, af, b2, b3);
                            }
                        }
                        orun[2 * xp][0] += oa[0] + oa[2];
                        orun[2 * xp][1] += oa[1] + oa[3];
                        if (2 * xp + 1 < kMaxNt / 2) {
                            orun[2 * xp + 1][0] += ob[0] + ob[2];
                            orun[2 * xp + 1][1] += ob[1] + ob[3];
                        }
                    }
                }
                l_run = l_run * a_run + l_seg * a_seg;
                m_run = m_new;
                // 5: clear the other parity's accumulator for the next segment
                {
                    float *vz = GB.va[pp ^ 1];
                    for (int x = phase * 32 + lane; x < 8 * D; x += grp_sz * 32) vz[x] = 0.f;
                }
                par[grp] = pp ^ 1;
                // 6: end of run -> write the record, ticket, maybe combine
                if (h[H_FLAGS] & kSegLastOfRun) {
                    const int recf = 8 * D + kRecFloatsExtra;
                    float *rec = p.rec + ((int64_t)h[H_REC] * p.nrg + rg) * recf;
#pragma unroll
                    for (int x = 0; x < kMaxNt / 2; ++x) {
                        const int ct = phase + x * grp_sz;
                        if (ct < kMaxNt) {
                            float2 v = make_float2(orun[x][0], orun[x][1]);
                            __stcg(reinterpret_cast<float2 *>(rec + quad * D + 8 * ct + 2 * qlane), v);
                        }
                    }
                    if (phase == 0 && qlane == 0) {
                        __stcg(rec + 8 * D + quad, m_run);
                        __stcg(rec + 8 * D + 8 + quad, l_run);
                    }
                    __threadfence();
                    if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                    if (phase == 0 && lane == 0) {
                        const uint32_t old = atomicAdd(&p.tickets[g * p.nrg + rg], 1u);
                        flags[grp] = (old == (uint32_t)expected_arrivals(p, g, rg) - 1) ? 1 : 0;
                    }
                    if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                    if (flags[grp]) {
                        __threadfence();
                        combine_rows<D>(p, g, rg, phase * 32 + lane, bar_n);
                        if (phase == 0 && lane == 0) p.tickets[g * p.nrg + rg] = 0u;
                    }
                }
            }
        } else if (kind == kTail) {
            // ---------------------------------------------- dense tail item
            const int i = h[H_QI], t0 = h[H_T0], t1 = h[H_T1], item = h[H_E];
            const int rgt = grp;
            const bool active = rgt < p.nrg_t;
            if (active) {
                const int pp = par[grp];
                const int rloc = 8 * rgt + quad;  // query head within the group
                const uint16_t *qrow = (rloc < p.G) ? p.q + ((int64_t)i * p.hq + g * p.G + rloc) * D : nullptr;
#pragma unroll
                for (int kc = 0; kc < kMaxKs; ++kc) {
                    qf[kc][0] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 2 * qlane) : 0u;
                    qf[kc][1] = 0u;
                    qf[kc][2] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + 16 * kc + 8 + 2 * qlane) : 0u;
                    qf[kc][3] = 0u;
                }
                m_w = -INFINITY;
                l_w = 0.f;
#pragma unroll
                for (int x = 0; x < kMaxNt; ++x) vacc[x][0] = vacc[x][1] = vacc[x][2] = vacc[x][3] = 0.f;
                constexpr uint32_t half = 64 * 64 * 2;
                const uint32_t kb = sbase, vb = sbase + (D / 64) * half;
                const int ntok = t1 - t0;
                const int nsub = (ntok + 15) / 16;
                for (int u = phase; u < nsub; u += grp_sz) {
                    const int tga = 2 * u, tgb = tga + 1;
                    float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
                    {
                        const int mi = lane / 8;
                        const int tr = 8 * ((mi < 2) ? tga : tgb) + (lane % 8);  // token row in the box
#pragma unroll
                        for (int kc = 0; kc < kMaxKs; ++kc) {
                            const int ch = 2 * kc + (mi & 1);
                            const uint32_t addr = kb + (ch / 8) * half + tr * 128 + (((ch % 8) ^ (tr % 8)) * 16);
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4(addr, b0, b1, b2, b3);
                            mma16816(sa, qf[kc], b0, b1);
                            mma16816(sb, qf[kc], b2, b3);
                        }
                    }
                    const int tl = 8 * tga + 2 * qlane;
                    float s0 = sa[0] * p.scale_log2, s1 = sa[1] * p.scale_log2;
                    float s2 = sb[0] * p.scale_log2, s3 = sb[1] * p.scale_log2;
                    if (tl >= ntok) s0 = -INFINITY;
                    if (tl + 1 >= ntok) s1 = -INFINITY;
                    if (tl + 8 >= ntok) s2 = -INFINITY;
                    if (tl + 9 >= ntok) s3 = -INFINITY;
                    const float mx = quad_max(fmaxf(fmaxf(s0, s1), fmaxf(s2, s3)));
                    if (mx > m_w + 8.f) {
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
                    {
                        const int mi = lane / 8;
                        const int tr = 8 * ((mi & 1) ? tgb : tga) + (lane % 8);
#pragma unroll
                        for (int cp = 0; cp < kMaxKs; ++cp) {
                            const int ch = 2 * cp + (mi >> 1);
                            const uint32_t addr = vb + (ch / 8) * half + tr * 128 + (((ch % 8) ^ (tr % 8)) * 16);
                            uint32_t b0, b1, b2, b3;
                            ldsm_x4_t(addr, b0, b1, b2, b3);
                            mma16816(vacc[2 * cp], pa, b0, b1);
                            mma16816(vacc[2 * cp + 1], pa, b2, b3);
                        }
                    }
                }
                // merge the group's warps; the merged accumulator is the output
                const float lq = quad_sum(l_w);
                if (qlane == 0) {
                    GB.ml[pp][(phase * 8 + quad) * 2 + 0] = m_w;
                    GB.ml[pp][(phase * 8 + quad) * 2 + 1] = lq;
                }
                if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                float m_seg = -INFINITY;
                for (int w = 0; w < grp_sz; ++w) m_seg = fmaxf(m_seg, GB.ml[pp][(w * 8 + quad) * 2]);
                float l_seg = 0.f;
                for (int w = 0; w < grp_sz; ++w)
                    l_seg += exp2_diff(GB.ml[pp][(w * 8 + quad) * 2], m_seg) * GB.ml[pp][(w * 8 + quad) * 2 + 1];
                const float sc = exp2_diff(m_w, m_seg);
                float *va = GB.va[pp];
                if (sc != 0.f) {
#pragma unroll
                    for (int x = 0; x < kMaxNt; ++x) {
                        const int c = 8 * x + 2 * qlane;
                        atomicAdd(&va[quad * D + c], (vacc[x][0] + vacc[x][2]) * sc);
                        atomicAdd(&va[quad * D + c + 1], (vacc[x][1] + vacc[x][3]) * sc);
                    }
                }
                if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                const int recf = 8 * D + kRecFloatsExtra;
                float *rec = p.rec + (p.tail_rec_base + (int64_t)item * p.nrg_t + rgt) * recf;
                for (int x = phase * 32 + lane; x < 8 * D / 4; x += grp_sz * 32)
                    __stcg(reinterpret_cast<float4 *>(rec) + x, reinterpret_cast<const float4 *>(va)[x]);
                if (phase == 0 && qlane == 0) {
                    __stcg(rec + 8 * D + quad, m_seg);
                    __stcg(rec + 8 * D + 8 + quad, l_seg);
                }
                {
                    float *vz = GB.va[pp ^ 1];
                    for (int x = phase * 32 + lane; x < 8 * D; x += grp_sz * 32) vz[x] = 0.f;
                }
                par[grp] = pp ^ 1;
                __threadfence();
                if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                // tickets of the prefix row groups these query rows belong to
                const int ra = i * p.G + 8 * rgt, rb = i * p.G + min(8 * rgt + 8, p.G);  // [ra, rb)
                for (int rg = ra / 8; rg <= (rb - 1) / 8; ++rg) {
                    if (phase == 0 && lane == 0) {
                        const uint32_t old = atomicAdd(&p.tickets[g * p.nrg + rg], 1u);
                        flags[grp] = (old == (uint32_t)expected_arrivals(p, g, rg) - 1) ? 1 : 0;
                    }
                    if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                    if (flags[grp]) {
                        __threadfence();
                        combine_rows<D>(p, g, rg, phase * 32 + lane, bar_n);
                        if (phase == 0 && lane == 0) p.tickets[g * p.nrg + rg] = 0u;
                    }
                    if (!group_sync(gbar, gph, bidx, lane, p.status)) return;
                }
            }
        }

        // release the slot (one arrival per consumer warp)
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars[kSlots + slot]));
    }
}

}  // namespace

int decode_smem_bytes(int head_dim, int nrg_cta)
{
    const int groups = max(nrg_cta, 4);
    return head_dim == 64 ? SmemLayout<64>::bytes(groups) : SmemLayout<128>::bytes(groups);
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
        cudaError_t e = which == 0
                            ? cudaFuncSetAttribute(decode_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes)
                            : cudaFuncSetAttribute(decode_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
        if (e != cudaSuccess) return e;
        configured[which] = smem_bytes;
    }
    if (which == 0) return cudaLaunchKernelEx(&cfg, decode_kernel<64>, p, mk, mv);
    return cudaLaunchKernelEx(&cfg, decode_kernel<128>, p, mk, mv);
}

}  // namespace milo
