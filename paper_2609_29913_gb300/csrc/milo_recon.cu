// milo_recon.cu -- reconstruct-then-attend: the paper's own inference path
// (Alg. 1 Stage 2 with the fused reconstruction of Sec. 3.5), kept beside the
// rank-space path as its comparison, and the path for factors of pre-RoPE
// keys (Sec. 3), whose rotation depends on each token's position and so
// cannot be moved into a shared projection.
//
// Work: the prefix is cut on the host into chunks of at most kRcChunkTiles
// tiles of kRcTok tokens of one entry (block b, KV head g); one thread block
// of 8 warps per (chunk, group of up to kRcRows query rows of KV head g).  Per
// tile the block
//   1. reconstructs the dense keys and values of the tile's tokens,
//        K^ = C^K P^K,  V^ = C^V P^V        (Eq. 3 with Sigma folded into C)
//      with mma.sync (bf16 factors, fp32 sums; warp w makes tokens
//      16 (w % 4) .. + 15 and half of the columns: the pairs (i, i + d/2) of
//      its half), rotates each key to its position when the plan holds
//      pre-RoPE factors, and stores both tiles in shared memory as fp16, as
//      the paper's kernel fills its fp16 KV buffer;
//   2. runs flash decoding over them (Eq. 1): scores q K^T, an online
//      softmax in log2 units, o += p V^ (fp16 operands, fp32 sums).  Each
//      16-row fragment of the group has W warps (4, 4, 2 or 1 for groups of
//      up to 16, 32, 64 or 128 rows), which split the tile's tokens and merge
//      at the end.
// Each (chunk, row group) then adds its (o, m, l) into the per-row
// accumulators of KV head g by the shared-reference merge of milo_merge.cuh
// (or lists a record for an outlier maximum), like every other item of a
// decode call; the call's dense-tail items run on the chunk grid before this
// grid and its finish grid after it.
//
// The factors stream through a ring of three tile buffers filled by 1-D bulk
// copies (one mbarrier each); P^K and P^V of the chunk's entry are copied
// once.  Every wait is bounded (~2 s) and sets MILO_ERR_TIMEOUT; a block that
// gives up waits (bounded) for its remaining copies and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "milo.h"
#include "milo_internal.h"
#include "milo_merge.cuh"
#include "milo_ptx.cuh"

namespace milo {
namespace {

constexpr int kRcWarps = 8;
constexpr int kRcThreads = 32 * kRcWarps;
constexpr int kRcRing = 3;

template <int D>
struct RcLay {
    static constexpr int kPHalf = D * D * 2;                 // P^K or P^V, up to D ranks (16-rank padded)
    static constexpr int kCSide = kRcTok * D * 2 + 128;      // C^K (or C^V) rows of one tile, + one core
    static constexpr int kCBuf = 2 * kCSide;                 // C^K then C^V
    static constexpr int kPK = 0;
    static constexpr int kPV = kPK + kPHalf;
    static constexpr int kC = kPV + kPHalf;                  // ring of kRcRing tile buffers
    static constexpr int kK = kC + kRcRing * kCBuf;          // K^ tile, fp16 cores [token group][column group]
    static constexpr int kV = kK + kRcTok * D * 2;           // V^ tile, same
    static constexpr int kBar = kV + kRcTok * D * 2;         // mbarriers: P, then the ring
    static constexpr int kTotal = kBar + 8 * (1 + kRcRing) + 16;
    // after the last tile the ring holds the warps' merge records:
    // [warp][D/8 column tiles][32 lanes] float4, then [warp][32 lanes] float4 (m0, m1, l0, l1)
    static constexpr int kXO = kC;
    static constexpr int kXM = kXO + kRcWarps * (D / 8) * 32 * 16;
    static_assert(kXM + kRcWarps * 32 * 16 <= kC + kRcRing * kCBuf, "merge records fit the ring");
    static_assert(kTotal <= 232448, "one block per SM");
};

// D(16x8 f32) += A(16x16 f16, row) * B(16x8 f16, col)
__device__ __forceinline__ void mma16816_f16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_half2(float x0, float x1)
{
    const __half2 h = __floats2half2_rn(x0, x1);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// bf16x2 bits -> f16x2 bits (exact for values inside the f16 range)
__device__ __forceinline__ uint32_t bf2_to_h2(uint32_t x)
{
    const float lo = __uint_as_float(x << 16), hi = __uint_as_float(x & 0xffff0000u);
    return pack_half2(lo, hi);
}

// The 8-column tiles of a warp's half h of the head dimension: local tile
// i < D/32 is column tile h D/32 + i, and local tile i + D/32 its rotary
// partner (the same columns + D/2).
template <int D>
__device__ __forceinline__ int col_tile(int h, int i)
{
    return i < D / 32 ? h * (D / 32) + i : D / 16 + h * (D / 32) + (i - D / 32);
}

// One fp32 tile of 16 tokens x half the columns (warp-fragment layout: local
// tile i, elements 0,1 row r4, columns 8 col_tile(h, i) + 2c4 + {0,1};
// elements 2,3 row r4 + 8) = C (16 tokens x rank, cores [token group][rank
// group], nr = rank groups) times P (rank x D, cores [rank group][column
// group]), over ks16 16-rank steps.  Rank groups past the rank read the
// zeroed rows of P.
template <int D>
__device__ __forceinline__ void reconstruct16(float (&acc)[D / 16][4], uint32_t c_base, int tg0, int nr, int ks16,
                                              uint32_t p_base, int h, int mi, int mr)
{
#pragma unroll
    for (int i = 0; i < D / 16; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
#pragma unroll 1
    for (int ks = 0; ks < ks16; ++ks) {
        uint32_t a[4];
        // matrices (tg0, 2ks), (tg0 + 1, 2ks), (tg0, 2ks + 1), (tg0 + 1, 2ks + 1)
        ldsm_x4(c_base + ((tg0 + (mi & 1)) * nr + 2 * ks + (mi >> 1)) * 128 + mr * 16, a[0], a[1], a[2], a[3]);
#pragma unroll
        for (int ip = 0; ip < D / 32; ++ip) {
            // transposed: (2ks, j), (2ks + 1, j), (2ks, j + 1), (2ks + 1, j + 1), j = col_tile(2 ip)
            const int j = col_tile<D>(h, 2 * ip);
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(p_base + ((2 * ks + (mi & 1)) * (D / 8) + j + (mi >> 1)) * 128 + mr * 16, b0, b1, b2, b3);
            mma16816(acc[2 * ip], a, b0, b1);
            mma16816(acc[2 * ip + 1], a, b2, b3);
        }
    }
}

// W warps per 16-row fragment (4, 2 or 1: groups of at most 32, 64 or 128
// rows); ROPE: the keys are pre-RoPE and turn to their positions.
template <int D, int W, bool ROPE>
__global__ void __launch_bounds__(kRcThreads, 1) recon_kernel(const __grid_constant__ DecodeParams p)
{
    using L = RcLay<D>;
    constexpr int NT = 8 / W;          // 8-token tiles of a warp's token slice
    constexpr int KD = D / 16;         // 16-wide steps over the head dimension
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int r4 = lane >> 2, c4 = lane & 3, mi = lane >> 3, mr = lane & 7;
    const uint32_t sbase = smem_u32(smem);
    const uint32_t bar_p = sbase + L::kBar;
    auto bar_c = [&](int k) { return bar_p + 8 * (1 + k % kRcRing); };

    const int nrgb = (p.rows_g + kRcRows - 1) / kRcRows;
    const int chunk = (int)blockIdx.x / nrgb, rgb = (int)blockIdx.x % nrgb;
    const int4 ck = p.rc_chunks[chunk];  // entry, first tile, tiles
    const EntryDev en = p.entries[ck.x];
    const int g = en.g, n = en.n;
    const int nrk = (en.rk + 7) >> 3, nrv = (en.rv + 7) >> 3;  // rank 8-groups
    const int tile0 = ck.y, ntiles = ck.z;
    const int n8 = (n + 7) & ~7;

    pdl_trigger();
    // zero everything the block reads: rank groups past a rank then meet zeros
    // in P, and token groups past the data finite values in C
    for (int i = tid; i < L::kBar / 16; i += kRcThreads) reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();

    auto issue_tile = [&](int k) {
        const uint32_t bar = bar_c(k), dst = sbase + L::kC + (k % kRcRing) * L::kCBuf;
        const int t0 = (tile0 + k) * kRcTok;
        const int rows8 = min(t0 + kRcTok, n8) - t0;
        const uint32_t kb = (uint32_t)rows8 * nrk * 16, vb = (uint32_t)rows8 * nrv * 16;
        mbar_arrive_tx(bar, kb + vb);
        if (kb) bulk_g2s(dst, p.packed + en.off_ck + (int64_t)t0 * nrk * 16, kb, bar);
        if (vb) bulk_g2s(dst + L::kCSide, p.packed + en.off_cv + (int64_t)t0 * nrv * 16, vb, bar);
    };
    if (tid == 0) {
        for (int i = 0; i < 1 + kRcRing; ++i) mbar_init(bar_p + 8 * i, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        const uint32_t pkb = (uint32_t)nrk * D * 16, pvb = (uint32_t)nrv * D * 16;
        mbar_arrive_tx(bar_p, pkb + pvb);
        if (pkb) bulk_g2s(sbase + L::kPK, p.packed + en.off_pk, pkb, bar_p);
        if (pvb) bulk_g2s(sbase + L::kPV, p.packed + en.off_pv, pvb, bar_p);
        for (int k = 0; k < min(ntiles, kRcRing); ++k) issue_tile(k);
    }
    __syncthreads();
    pdl_wait();  // q and the accumulators belong to the preceding grids until here

    // this warp's fragment (16 rows) and token slice
    const int frag = warp / W, slice = warp % W;
    const int rbase = rgb * kRcRows + 16 * frag;  // first row of the fragment within KV head g
    const bool frag_ok = rbase < p.rows_g;
    const int row0 = rbase + r4, row1 = row0 + 8;
    const bool ok0 = row0 < p.rows_g, ok1 = row1 < p.rows_g;
    // q rows as fp16 A fragments over the head dimension
    uint32_t qa[KD][4];
    {
        const uint16_t *q0 = p.q + ((int64_t)(row0 / p.G) * p.hq + g * p.G + row0 % p.G) * D + 2 * c4;
        const uint16_t *q1 = p.q + ((int64_t)(row1 / p.G) * p.hq + g * p.G + row1 % p.G) * D + 2 * c4;
#pragma unroll
        for (int ks = 0; ks < KD; ++ks) {
            const uint32_t x0 = ok0 ? *reinterpret_cast<const uint32_t *>(q0 + 16 * ks) : 0u;
            const uint32_t x1 = ok1 ? *reinterpret_cast<const uint32_t *>(q1 + 16 * ks) : 0u;
            const uint32_t x2 = ok0 ? *reinterpret_cast<const uint32_t *>(q0 + 16 * ks + 8) : 0u;
            const uint32_t x3 = ok1 ? *reinterpret_cast<const uint32_t *>(q1 + 16 * ks + 8) : 0u;
            qa[ks][0] = bf2_to_h2(x0);
            qa[ks][1] = bf2_to_h2(x1);
            qa[ks][2] = bf2_to_h2(x2);
            qa[ks][3] = bf2_to_h2(x3);
        }
    }
    float o[D / 8][4];
#pragma unroll
    for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    uint32_t ref0 = 0u, ref1 = 0u;

    bool ok = mbar_wait(bar_p, 0, p.status);
    ok = __syncthreads_and(ok);
    const uint32_t sK = sbase + L::kK, sV = sbase + L::kV;
    const int b = ck.x / p.hkv;
    int issued = min(ntiles, kRcRing);
    int landed = 0;  // tiles [0, landed) have been waited for
#pragma unroll 1
    for (int k = 0; ok && k < ntiles; ++k) {
        if (tid == 0 && k >= 1 && issued < ntiles) issue_tile(issued++);  // into the buffer tile k - 1 left
        ok = __syncthreads_and(mbar_wait(bar_c(k), (k / kRcRing) & 1, p.status));
        if (!ok) break;
        landed = k + 1;
        const uint32_t cb = sbase + L::kC + (k % kRcRing) * L::kCBuf;
        const int nv = min(kRcTok, n - (tile0 + k) * kRcTok);  // valid tokens of the tile

        // ---- 1. reconstruct 16 tokens x half of the columns (warp) of K^ and
        // V^ into fp16 tiles
        {
            const int mt = warp & 3, hh = warp >> 2;  // token 16-group, column half
            float acc[D / 16][4];
            reconstruct16<D>(acc, cb, 2 * mt, nrk, (nrk + 1) >> 1, sbase + L::kPK, hh, mi, mr);
            if constexpr (ROPE) {
                // pair (i, i + D/2) = local tiles (t, t + D/32), same registers;
                // angle = (tile start + u) theta_i from the plan's tables
                const float2 *tab_t = p.rope_tile + ((int64_t)p.rope_tile_base[b] + tile0 + k) * (D / 2);
#pragma unroll
                for (int t = 0; t < D / 32; ++t)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int i = 8 * col_tile<D>(hh, t) + 2 * c4 + (e & 1);
                        const int u = 16 * mt + r4 + (e >> 1) * 8;
                        const float2 a = __ldg(tab_t + i), c = __ldg(p.rope_off + u * (D / 2) + i);
                        const float cs = a.x * c.x - a.y * c.y, sn = a.y * c.x + a.x * c.y;
                        const float x0 = acc[t][e], x1 = acc[t + D / 32][e];
                        acc[t][e] = x0 * cs - x1 * sn;
                        acc[t + D / 32][e] = x1 * cs + x0 * sn;
                    }
            }
            uint32_t *kk = reinterpret_cast<uint32_t *>(smem + L::kK);
#pragma unroll
            for (int t = 0; t < D / 16; ++t) {
                const int j = col_tile<D>(hh, t);
                kk[((2 * mt) * (D / 8) + j) * 32 + r4 * 4 + c4] = pack_half2(acc[t][0], acc[t][1]);
                kk[((2 * mt + 1) * (D / 8) + j) * 32 + r4 * 4 + c4] = pack_half2(acc[t][2], acc[t][3]);
            }
            reconstruct16<D>(acc, cb + L::kCSide, 2 * mt, nrv, (nrv + 1) >> 1, sbase + L::kPV, hh, mi, mr);
            uint32_t *vv = reinterpret_cast<uint32_t *>(smem + L::kV);
#pragma unroll
            for (int t = 0; t < D / 16; ++t) {
                const int j = col_tile<D>(hh, t);
                vv[((2 * mt) * (D / 8) + j) * 32 + r4 * 4 + c4] = pack_half2(acc[t][0], acc[t][1]);
                vv[((2 * mt + 1) * (D / 8) + j) * 32 + r4 * 4 + c4] = pack_half2(acc[t][2], acc[t][3]);
            }
        }
        __syncthreads();

        // ---- 2. flash decoding of the fragment's rows over the warp's token slice
        if (frag_ok) {
            const int tg0 = slice * NT;  // first 8-token group of the slice
            float s[NT][4];
#pragma unroll
            for (int t = 0; t < NT; ++t) s[t][0] = s[t][1] = s[t][2] = s[t][3] = 0.f;
#pragma unroll
            for (int ks = 0; ks < KD; ++ks)
#pragma unroll
                for (int tp = 0; tp < NT / 2; ++tp) {
                    // matrices (tg, 2ks), (tg, 2ks + 1), (tg + 1, 2ks), (tg + 1, 2ks + 1)
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(sK + ((tg0 + 2 * tp + (mi >> 1)) * (D / 8) + 2 * ks + (mi & 1)) * 128 + mr * 16, b0, b1,
                            b2, b3);
                    mma16816_f16(s[2 * tp], qa[ks], b0, b1);
                    mma16816_f16(s[2 * tp + 1], qa[ks], b2, b3);
                }
            float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
            for (int t = 0; t < NT; ++t)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int tok = 8 * (tg0 + t) + 2 * c4 + (e & 1);
                    s[t][e] = tok < nv ? s[t][e] * p.scale_log2 : -INFINITY;
                }
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                mx0 = fmaxf(mx0, fmaxf(s[t][0], s[t][1]));
                mx1 = fmaxf(mx1, fmaxf(s[t][2], s[t][3]));
            }
            mx0 = quad_max(mx0);
            mx1 = quad_max(mx1);
            const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
            const float base0 = mn0 == -INFINITY ? 0.f : mn0, base1 = mn1 == -INFINITY ? 0.f : mn1;
            const float al0 = m0 == -INFINITY ? 0.f : ex2_approx(m0 - base0);
            const float al1 = m1 == -INFINITY ? 0.f : ex2_approx(m1 - base1);
            m0 = mn0;
            m1 = mn1;
            float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                s[t][0] = ex2_approx(s[t][0] - base0);
                s[t][1] = ex2_approx(s[t][1] - base0);
                s[t][2] = ex2_approx(s[t][2] - base1);
                s[t][3] = ex2_approx(s[t][3] - base1);
                ps0 += s[t][0] + s[t][1];
                ps1 += s[t][2] + s[t][3];
            }
            l0 = l0 * al0 + ps0;
            l1 = l1 * al1 + ps1;
#pragma unroll
            for (int j = 0; j < D / 8; ++j) {
                o[j][0] *= al0;
                o[j][1] *= al0;
                o[j][2] *= al1;
                o[j][3] *= al1;
            }
#pragma unroll
            for (int kk = 0; kk < NT / 2; ++kk) {
                const uint32_t a[4] = {pack_half2(s[2 * kk][0], s[2 * kk][1]), pack_half2(s[2 * kk][2], s[2 * kk][3]),
                                       pack_half2(s[2 * kk + 1][0], s[2 * kk + 1][1]),
                                       pack_half2(s[2 * kk + 1][2], s[2 * kk + 1][3])};
#pragma unroll
                for (int jp = 0; jp < D / 16; ++jp) {
                    // transposed: (tg, 2jp), (tg + 1, 2jp), (tg, 2jp + 1), (tg + 1, 2jp + 1)
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_t(sV + ((tg0 + 2 * kk + (mi & 1)) * (D / 8) + 2 * jp + (mi >> 1)) * 128 + mr * 16, b0, b1,
                              b2, b3);
                    mma16816_f16(o[2 * jp], a, b0, b1);
                    mma16816_f16(o[2 * jp + 1], a, b2, b3);
                }
            }
            // the first slice of a fragment sets or reads its rows' references
            // once it has a maximum (the result is used at the end)
            if (k == 0 && slice == 0) {
                ref0 = __shfl_sync(0xffffffffu, publish_ref(p, g, row0, ok0, c4, m0), lane & ~3);
                ref1 = __shfl_sync(0xffffffffu, publish_ref(p, g, row1, ok1, c4, m1), lane & ~3);
            }
        }
        __syncthreads();  // the K^ and V^ tiles are rewritten by the next tile
    }
    if (!ok) {
        // give up: let the copies still in flight land before the block exits
        if (tid == 0)
            for (int k = landed; k < issued; ++k) mbar_wait(bar_c(k), (k / kRcRing) & 1, p.status);
        return;
    }

    l0 = quad_sum(l0);
    l1 = quad_sum(l1);
    if constexpr (W > 1) {
        // the warps of a fragment merge through the ring (no copy in flight)
        float4 *xo = reinterpret_cast<float4 *>(smem + L::kXO);
        float4 *xm = reinterpret_cast<float4 *>(smem + L::kXM);
        if (slice != 0) {
#pragma unroll
            for (int j = 0; j < D / 8; ++j) xo[(warp * (D / 8) + j) * 32 + lane] = make_float4(o[j][0], o[j][1], o[j][2], o[j][3]);
            xm[warp * 32 + lane] = make_float4(m0, m1, l0, l1);
        }
        __syncthreads();
        if (slice == 0 && frag_ok) {
            float M0 = m0, M1 = m1;
#pragma unroll
            for (int s2 = 1; s2 < W; ++s2) {
                const float4 x = xm[(warp + s2) * 32 + lane];
                M0 = fmaxf(M0, x.x);
                M1 = fmaxf(M1, x.y);
            }
            // slice 0 always holds a token, so M0 and M1 are finite
            const float f00 = ex2_approx(m0 - M0), f01 = ex2_approx(m1 - M1);
            l0 *= f00;
            l1 *= f01;
#pragma unroll
            for (int j = 0; j < D / 8; ++j) {
                o[j][0] *= f00;
                o[j][1] *= f00;
                o[j][2] *= f01;
                o[j][3] *= f01;
            }
#pragma unroll
            for (int s2 = 1; s2 < W; ++s2) {
                const float4 x = xm[(warp + s2) * 32 + lane];
                const float f0 = x.x == -INFINITY ? 0.f : ex2_approx(x.x - M0);
                const float f1 = x.y == -INFINITY ? 0.f : ex2_approx(x.y - M1);
                l0 += f0 * x.z;
                l1 += f1 * x.w;
#pragma unroll
                for (int j = 0; j < D / 8; ++j) {
                    const float4 y = xo[((warp + s2) * (D / 8) + j) * 32 + lane];
                    o[j][0] += f0 * y.x;
                    o[j][1] += f0 * y.y;
                    o[j][2] += f1 * y.z;
                    o[j][3] += f1 * y.w;
                }
            }
            m0 = M0;
            m1 = M1;
        }
    }
    if (slice != 0 || !frag_ok) return;

    // ---- the (chunk, fragment) result into the accumulators of KV head g,
    // per group of 8 rows: rows r4 (group 2 frag) and r4 + 8 (group 2 frag + 1)
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const int row = half ? row1 : row0;
        const bool row_ok = half ? ok1 : ok0;
        const float m = half ? m1 : m0, l = half ? l1 : l0;
        const uint32_t refb = half ? ref1 : ref0;
        const float Mref = refb ? ref_dec(refb) : m;
        const bool direct = !__any_sync(0xffffffffu, row_ok && m - Mref > kDirectMax);
        const int rgg = rbase / 8 + half;
        const int64_t rec_idx = (int64_t)chunk * p.nrg + rgg;
        if (direct) {
            if (row_ok) {
                const float f = ex2_approx(m - Mref);
                float *orow = p.acc_o + ((int64_t)g * p.rows_max + row) * D + 2 * c4;
#pragma unroll
                for (int j = 0; j < D / 8; ++j)
                    atomicAdd(reinterpret_cast<float2 *>(orow + 8 * j),
                              make_float2(f * o[j][2 * half], f * o[j][2 * half + 1]));
                if (c4 == 0) atomicAdd(p.acc_l + (int64_t)g * p.rows_max + row, f * l);
            }
        } else {
            float *rec = p.rec + rec_idx * (8 * D + kRecFloatsExtra);
#pragma unroll
            for (int j = 0; j < D / 8; ++j)
                __stcg(reinterpret_cast<float2 *>(rec + r4 * D + 8 * j + 2 * c4),
                       make_float2(o[j][2 * half], o[j][2 * half + 1]));
            if (c4 == 0) {
                __stcg(rec + 8 * D + r4, m);
                __stcg(rec + 8 * D + 8 + r4, l);
            }
            if (lane == 0) {
                const int gr = g * p.nrg + rgg;
                const uint32_t kx = atomicAdd(p.ovf_cnt + gr, 1u);
                __stcg(reinterpret_cast<int4 *>(p.ovf_list) + (int64_t)gr * p.list_cap + kx,
                       make_int4((int)rec_idx, 8 * rgg, min(8, p.rows_g - 8 * rgg), 0));
            }
        }
    }
}

template <int D, int W, bool ROPE>
cudaError_t launch_one(const DecodeParams &p, int blocks, cudaStream_t stream)
{
    static bool configured[kMaxDevices] = {};
    const int dev = attribute_slot();
    if (dev < 0 || !configured[dev]) {
        cudaError_t e = cudaFuncSetAttribute(recon_kernel<D, W, ROPE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             RcLay<D>::kTotal);
        if (e != cudaSuccess) return e;
        if (dev >= 0) configured[dev] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks);
    cfg.blockDim = dim3(kRcThreads);
    cfg.dynamicSmemBytes = (size_t)RcLay<D>::kTotal;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, recon_kernel<D, W, ROPE>, p);
}

template <int D, bool ROPE>
cudaError_t launch_d(const DecodeParams &p, int blocks, int w, cudaStream_t stream)
{
    return w == 4 ? launch_one<D, 4, ROPE>(p, blocks, stream)
           : w == 2 ? launch_one<D, 2, ROPE>(p, blocks, stream)
                    : launch_one<D, 1, ROPE>(p, blocks, stream);
}

}  // namespace

cudaError_t launch_recon(const DecodeParams &p, int num_chunks, cudaStream_t stream)
{
    const int64_t blocks = (int64_t)num_chunks * ((p.rows_g + kRcRows - 1) / kRcRows);
    if (blocks < 1 || blocks > 0x7fffffff) return cudaErrorInvalidValue;
    // warps per 16-row fragment: groups of up to 32 rows (one or two
    // fragments) give each fragment 4 warps, of up to 64 rows 2, else 1
    const int f = ((p.rows_g < kRcRows ? p.rows_g : kRcRows) + 15) / 16;
    const int w = f <= 2 ? 4 : f <= 4 ? 2 : 1;
    const bool rope = p.rope_tile != nullptr;
    if (p.d == 64) return rope ? launch_d<64, true>(p, (int)blocks, w, stream) : launch_d<64, false>(p, (int)blocks, w, stream);
    return rope ? launch_d<128, true>(p, (int)blocks, w, stream) : launch_d<128, false>(p, (int)blocks, w, stream);
}

}  // namespace milo
