// milo_chunk.cu -- the split-K decode of milo_decode.cu for up to 8 query rows
// per KV head (batch x heads of one KV head <= 8): one warp per chunk, many
// chunks per SM, each chunk streamed through two shared-memory slots.
//
// A chunk is a token range of one prefix entry (block b, KV head g).  Its warp
// walks a fixed sequence of pieces, each at most kPieceBytes and brought by
// bulk copies into one of two slots while the warp works on the other:
//
//   P^K pieces   q~ = scale * log2(e) * P^K q for up to 64 ranks per piece
//                (Eq. 3 folded into Eq. 1); q~ is kept as bf16 hi + lo rows of
//                the score A operand.
//   C pieces     whole 32-token tiles (C^K rows, then C^V rows of the same
//                tokens): scores s = C^K q~, an online softmax with a lazily
//                raised reference max, rank-space values v~ += C^V^T p.
//   P^V pieces   o += P^V^T v~ over up to 64 ranks per piece (Alg. 1 Stage
//                2's back-projection), v~ taken straight from the registers.
//
// The chunk's record is (o, max, sum) per query row.  The last chunk block
// of a prefix entry (a per-entry counter) merges the entry's chunk records
// into one entry record; an entry of one chunk writes its entry record
// directly.  Entry and tail records are counted per KV head.  A dense-tail item (one
// query's tail split for one KV head, kTailTokens tokens) brings its K and V
// rows with 3-D TMA boxes (8 head dimensions x kTailTokens rows each, landing
// as cores [column group][token group]) and runs the C steps on them with
// q~ = scale * log2(e) * q; its values are already o.  The
// last thread blocks of the grid merge: one warp per (KV head, row, quarter
// of the head dimension) waits (bounded) until every entry and tail record
// of its KV head is counted, then combines them with the log-sum-exp rule (Eq. 1 over a
// partition of the tokens) and writes the output; the last of a KV head's
// merge blocks resets its counters for the next call.  Chunk and tail blocks
// never wait on other blocks, and they come first in the grid.
//
// Shared-memory cores are 8 rows x 16 bytes (rows = tokens or ranks); a core
// past the data reads a zero line, so no product meets stale memory.  Every
// wait is bounded (~2 s) and sets MILO_ERR_TIMEOUT.
#include <cuda.h>
#include <cuda_bf16.h>

#include <type_traits>

#include "milo.h"
#include "milo_internal.h"
#include "milo_ptx.cuh"

namespace milo {
namespace {

constexpr int kPieceBytes = 16384;  // one slot
constexpr int kTile = 32;           // tokens per tile

template <int D>
struct CLay {
    static constexpr int kQ = 2 * kPieceBytes;                  // q~ A fragments [D/16][32 lanes][4]
    static constexpr int kZero = kQ + (D / 16) * 32 * 16;       // a zero core line
    static constexpr int kBar = kZero + 128;                    // 2 mbarriers
    static constexpr int kTotal = kBar + 16;
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
    s.rpp = CLay<D>::kRanksPerPiece / 8;
    s.npk = (c.nrk + s.rpp - 1) / s.rpp;
    s.npv = (c.nrv + s.rpp - 1) / s.rpp;
    s.tpp = max(1, kPieceBytes / (kTile * (c.nrk + c.nrv) * 16));
    s.nc = (c.ntok + s.tpp * kTile - 1) / (s.tpp * kTile);
    return s;
}

constexpr int kMergeWarpsPerHead = 32;  // 8 rows x 4 quarters of the head dimension

// This block's record is written: count it for KV head g (lane 0 after a fence).
__device__ __forceinline__ void count_record(const DecodeParams &p, int g, int lane)
{
    __threadfence();
    __syncwarp();
    if (lane == 0) atomicAdd(&p.head_cnt[g], 1u);
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *ptr)
{
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ptr) : "memory");
    return v;
}

// The last chunk of a prefix entry: merge the entry's nch chunk records
// (c0 ...) into its entry record.  Lane l: row l / 4, quarter l % 4.
template <int D>
__device__ void merge_entry(const DecodeParams &p, int c0, int nch, float *dst, int lane)
{
    constexpr int kF4 = D / 16;
    constexpr int kLoads = 4;
    const int recf = 8 * D + kRecFloatsExtra;
    const int row = lane >> 2, qq = lane & 3;
    float M = -INFINITY, Lsum = 0.f;
    float4 acc[kF4];
#pragma unroll
    for (int f = 0; f < kF4; ++f) acc[f] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s0 = 0; s0 < nch; s0 += kLoads) {
        float mm[kLoads], ll[kLoads];
        float4 oo[kLoads][kF4];
#pragma unroll
        for (int j = 0; j < kLoads; ++j) {
            mm[j] = -INFINITY;
            ll[j] = 0.f;
#pragma unroll
            for (int f = 0; f < kF4; ++f) oo[j][f] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (s0 + j < nch) {
                const float *r = p.rec + (int64_t)(c0 + s0 + j) * recf;
                mm[j] = __ldcg(r + 8 * D + row);
                ll[j] = __ldcg(r + 8 * D + 8 + row);
#pragma unroll
                for (int f = 0; f < kF4; ++f)
                    oo[j][f] = __ldcg(reinterpret_cast<const float4 *>(r + row * D + qq * (D / 4)) + f);
            }
        }
        float Mc = M;
#pragma unroll
        for (int j = 0; j < kLoads; ++j) Mc = fmaxf(Mc, mm[j]);
        const float a = exp2_diff(M, Mc);
        Lsum *= a;
#pragma unroll
        for (int f = 0; f < kF4; ++f) {
            acc[f].x *= a; acc[f].y *= a; acc[f].z *= a; acc[f].w *= a;
        }
#pragma unroll
        for (int j = 0; j < kLoads; ++j) {
            const float w = exp2_diff(mm[j], Mc);
            Lsum += w * ll[j];
#pragma unroll
            for (int f = 0; f < kF4; ++f) {
                acc[f].x += w * oo[j][f].x; acc[f].y += w * oo[j][f].y;
                acc[f].z += w * oo[j][f].z; acc[f].w += w * oo[j][f].w;
            }
        }
        M = Mc;
    }
#pragma unroll
    for (int f = 0; f < kF4; ++f) __stcg(reinterpret_cast<float4 *>(dst + row * D + qq * (D / 4)) + f, acc[f]);
    if (qq == 0) {
        __stcg(dst + 8 * D + row, M);
        __stcg(dst + 8 * D + 8 + row, Lsum);
    }
}

// One merge warp: KV head g, row k of the row group, quarter qq of the head
// dimension.  Lane l takes records l, l + 32, ...; the 32 partial merges meet
// through a shuffle butterfly.
template <int D>
__device__ void merge_warp(const DecodeParams &p, int mb, int lane)
{
    constexpr int kF4 = D / 16;  // float4 columns per quarter
    constexpr int kChunkLoads = 4;
    const int g = mb / kMergeWarpsPerHead, k = (mb / 4) % 8, qq = mb % 4;
    const int recf = 8 * D + kRecFloatsExtra;
    const int gs0 = p.g_entry_begin[g], nprefix = p.g_entry_begin[g + 1] - gs0;
    const int S = p.tail_splits, nsrc = nprefix + p.batch * S;
    pdl_wait();  // the output belongs to the preceding grids until here
    // every record of KV head g: its chunks and the tail items of every query
    if (lane == 0) {
        const uint64_t t0 = globaltimer();
        while (ld_acquire(&p.head_cnt[g]) < (uint32_t)nsrc) {
            __nanosleep(200);
            if (globaltimer() - t0 > kTimeoutNs) {
                atomicCAS(p.status, 0, (int32_t)MILO_ERR_TIMEOUT);
                break;
            }
        }
    }
    __syncwarp();
    const bool row_ok = k < p.rows_g;
    if (row_ok) {
        const int i = k / p.G, hh = k % p.G;
        const float *tail0 = p.rec + (p.tail_rec_base + (int64_t)(i * p.hkv + g) * S) * recf;
        const int ns = nprefix + S;  // this row: the prefix chunks and query i's tail splits
        float M = -INFINITY, Lsum = 0.f;
        float4 acc[kF4];
#pragma unroll
        for (int j = 0; j < kF4; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s0 = lane; s0 < ns; s0 += 32 * kChunkLoads) {
            float mm[kChunkLoads], ll[kChunkLoads];
            float4 oo[kChunkLoads][kF4];
#pragma unroll
            for (int j = 0; j < kChunkLoads; ++j) {
                const int s = s0 + 32 * j;
                mm[j] = -INFINITY;
                ll[j] = 0.f;
#pragma unroll
                for (int f = 0; f < kF4; ++f) oo[j][f] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (s < ns) {
                    const bool pre = s < nprefix;
                    const int row = pre ? k : hh;
                    const float *r = pre ? p.rec + (int64_t)(gs0 + s) * recf : tail0 + (int64_t)(s - nprefix) * recf;
                    mm[j] = __ldcg(r + 8 * D + row);
                    ll[j] = __ldcg(r + 8 * D + 8 + row);
#pragma unroll
                    for (int f = 0; f < kF4; ++f)
                        oo[j][f] = __ldcg(reinterpret_cast<const float4 *>(r + row * D + qq * (D / 4)) + f);
                }
            }
            float Mc = M;
#pragma unroll
            for (int j = 0; j < kChunkLoads; ++j) Mc = fmaxf(Mc, mm[j]);
            const float a = exp2_diff(M, Mc);
            Lsum *= a;
#pragma unroll
            for (int f = 0; f < kF4; ++f) {
                acc[f].x *= a; acc[f].y *= a; acc[f].z *= a; acc[f].w *= a;
            }
#pragma unroll
            for (int j = 0; j < kChunkLoads; ++j) {
                const float w = exp2_diff(mm[j], Mc);
                Lsum += w * ll[j];
#pragma unroll
                for (int f = 0; f < kF4; ++f) {
                    acc[f].x += w * oo[j][f].x; acc[f].y += w * oo[j][f].y;
                    acc[f].z += w * oo[j][f].z; acc[f].w += w * oo[j][f].w;
                }
            }
            M = Mc;
        }
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float Mo = __shfl_xor_sync(0xffffffffu, M, off);
            const float Lo = __shfl_xor_sync(0xffffffffu, Lsum, off);
            const float Mn = fmaxf(M, Mo);
            const float a = exp2_diff(M, Mn), b = exp2_diff(Mo, Mn);
            Lsum = Lsum * a + Lo * b;
#pragma unroll
            for (int f = 0; f < kF4; ++f) {
                const float4 o2 = make_float4(__shfl_xor_sync(0xffffffffu, acc[f].x, off),
                                              __shfl_xor_sync(0xffffffffu, acc[f].y, off),
                                              __shfl_xor_sync(0xffffffffu, acc[f].z, off),
                                              __shfl_xor_sync(0xffffffffu, acc[f].w, off));
                acc[f] = make_float4(acc[f].x * a + o2.x * b, acc[f].y * a + o2.y * b, acc[f].z * a + o2.z * b,
                                     acc[f].w * a + o2.w * b);
            }
            M = Mn;
        }
        const float inv = 1.f / Lsum;
        float *dst = p.out + ((int64_t)i * p.hq + g * p.G + hh) * D + qq * (D / 4);
#pragma unroll
        for (int f = 0; f < kF4; ++f)
            if (lane == f)
                reinterpret_cast<float4 *>(dst)[f] =
                    make_float4(acc[f].x * inv, acc[f].y * inv, acc[f].z * inv, acc[f].w * inv);
    }
    // the last merge warp of KV head g resets its counters for the next call
    __syncwarp();
    if (lane == 0 && atomicAdd(&p.head_cnt[p.hkv + g], 1u) == kMergeWarpsPerHead - 1) {
        p.head_cnt[g] = 0u;
        p.head_cnt[p.hkv + g] = 0u;
        __threadfence();
    }
}

template <int D>
__global__ void __launch_bounds__(32)
    chunk_kernel(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tmap_k,
                 const __grid_constant__ CUtensorMap tmap_v)
{
    static_assert(2 * (D / 8) * kTailTokens * 16 <= 2 * kPieceBytes, "a tail item fits the two slots");
    using L = CLay<D>;
    constexpr int KD = D / 16;  // 16-wide k-steps over the head dimension
    constexpr int NT = D / 8;   // 8-wide tiles over the head dimension (and the largest rank)
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x;
    const int r4 = lane >> 2, c4 = lane & 3;  // mma fragment row and column pair
    const int mi = lane >> 3, mr = lane & 7;  // ldmatrix: matrix and row this lane addresses
    uint4 *sq = reinterpret_cast<uint4 *>(smem + L::kQ);
    const uint32_t zline = smem_u32(smem + L::kZero) + mr * 16;
    const uint32_t bar0 = smem_u32(smem + L::kBar);
    const int recf = 8 * D + kRecFloatsExtra;
    const bool is_tail = (int)blockIdx.x >= p.num_chunks;

    pdl_trigger();
    const int first_merge = p.num_chunks + (p.has_tail ? p.num_tail_items : 0);
    if ((int)blockIdx.x >= first_merge) {
        merge_warp<D>(p, (int)blockIdx.x - first_merge, lane);
        return;
    }
    for (int i = lane; i < (L::kBar - L::kQ) / 16; i += 32)
        reinterpret_cast<uint4 *>(smem + L::kQ)[i] = make_uint4(0u, 0u, 0u, 0u);

    ChunkDev ch = {};
    Pieces ps = {};
    int g = 0, ntok = 0, nrk = 0, nrv = 0;
    if (!is_tail) {
        ch = p.chunks[blockIdx.x];
        ps = pieces_of<D>(ch);
        g = ch.g;
        ntok = ch.ntok;
        nrk = ch.nrk;
        nrv = ch.nrv;
    }
    // piece k into slot k & 1 (lane 0)
    auto issue = [&](int k) {
        const uint32_t bar = bar0 + 8 * (k & 1), dst = smem_u32(smem) + (k & 1) * kPieceBytes;
        if (k < ps.npk) {
            const int r0 = k * ps.rpp, r1 = min(r0 + ps.rpp, ch.nrk);
            const uint32_t b = (uint32_t)(r1 - r0) * D * 16;
            mbar_arrive_tx(bar, b);
            bulk_g2s(dst, p.packed + ch.pk + (int64_t)r0 * D * 16, b, bar);
        } else if (k < ps.npk + ps.nc) {
            const int t0 = (k - ps.npk) * ps.tpp * kTile;
            const int r8 = min(t0 + ps.tpp * kTile, ch.tok8) - t0;  // rows (a multiple of 8)
            const uint32_t kb = (uint32_t)r8 * ch.nrk * 16, vb = (uint32_t)r8 * ch.nrv * 16;
            mbar_arrive_tx(bar, kb + vb);
            bulk_g2s(dst, p.packed + ch.ck + (int64_t)t0 * ch.nrk * 16, kb, bar);
            bulk_g2s(dst + kb, p.packed + ch.cv + (int64_t)t0 * ch.nrv * 16, vb, bar);
        } else {
            const int r0 = (k - ps.npk - ps.nc) * ps.rpp, r1 = min(r0 + ps.rpp, ch.nrv);
            const uint32_t b = (uint32_t)(r1 - r0) * D * 16;
            mbar_arrive_tx(bar, b);
            bulk_g2s(dst, p.packed + ch.pv + (int64_t)r0 * D * 16, b, bar);
        }
    };
    if (lane == 0) {
        mbar_init(bar0, 1);
        mbar_init(bar0 + 8, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (!is_tail) {
            issue(0);
            if (ps.total() > 1) issue(1);
        }
    }
    __syncwarp();
    pdl_wait();  // q, the tails and the records belong to the preceding grids until here

    // the warp's online-softmax state and rank-space values
    float m_w = -INFINITY, l_w = 0.f;
    float vacc[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n) vacc[n][0] = vacc[n][1] = vacc[n][2] = vacc[n][3] = 0.f;

    // One 32-token tile at token tb of the tile data: C^K core (tg, rg) at
    // kb + tg * ktg + rg * krg, C^V core at vb + tg * vtg + rg * vrg; tg8 token
    // groups present, tokens < nv valid.  R16 (a compile-time constant, at
    // least both ranks / 16) fixes the 16-rank steps, so that the body is one
    // straight block; rank groups past a rank and token groups past the data
    // read the zero line.
    auto tile = [&](auto r16c, uint32_t kb, uint32_t ktg, uint32_t krg, uint32_t vb, uint32_t vtg, uint32_t vrg,
                    int tb, int tg8, int nv) {
        constexpr int R16 = decltype(r16c)::value;
        float s4[4][4];
#pragma unroll
        for (int n = 0; n < 4; ++n) s4[n][0] = s4[n][1] = s4[n][2] = s4[n][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < R16; ++ks) {
            const uint4 q4 = sq[ks * 32 + lane];
            const uint32_t qa[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                // matrices: (tg0, 2ks), (tg0, 2ks + 1), (tg0 + 1, 2ks), (tg0 + 1, 2ks + 1)
                const int tg = tb / 8 + 2 * h + (mi >> 1), rg = 2 * ks + (mi & 1);
                const uint32_t addr = (tg < tg8 && rg < nrk) ? kb + tg * ktg + rg * krg + mr * 16 : zline;
                uint32_t b0, b1, b2, b3;
                ldsm_x4(addr, b0, b1, b2, b3);
                mma16816(s4[2 * h], qa, b0, b1);
                mma16816(s4[2 * h + 1], qa, b2, b3);
            }
        }
        // score of token tb + 8n + 2 c4 + j: hi rows + lo rows
        float sv8[8];
#pragma unroll
        for (int n = 0; n < 4; ++n) {
            const int tok = tb + 8 * n + 2 * c4;
            sv8[2 * n] = tok < nv ? s4[n][0] + s4[n][2] : -INFINITY;
            sv8[2 * n + 1] = tok + 1 < nv ? s4[n][1] + s4[n][3] : -INFINITY;
        }
        const float lm = fmaxf(fmaxf(fmaxf(sv8[0], sv8[1]), fmaxf(sv8[2], sv8[3])),
                               fmaxf(fmaxf(sv8[4], sv8[5]), fmaxf(sv8[6], sv8[7])));
        // lazy rescale (p stays <= 2^8): the row maximum is formed only when
        // some score passes the reference by more than 8
        if (__any_sync(0xffffffffu, lm > m_w + 8.f)) {
            const float mx = quad_max(lm);
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
        float pr[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) pr[j] = exp2_diff(sv8[j], m_w);
        l_w += ((pr[0] + pr[1]) + (pr[2] + pr[3])) + ((pr[4] + pr[5]) + (pr[6] + pr[7]));
        // A fragments of p for the two 16-token halves (rows 0-7 hi, 8-15 lo)
        uint32_t pa[2][4];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            split_hi_lo(pr[4 * h], pr[4 * h + 1], pa[h][0], pa[h][1]);
            split_hi_lo(pr[4 * h + 2], pr[4 * h + 3], pa[h][2], pa[h][3]);
        }
#pragma unroll
        for (int jp = 0; jp < R16; ++jp) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                // matrices (transposed): (tg0, 2jp), (tg0 + 1, 2jp), (tg0, 2jp + 1), (tg0 + 1, 2jp + 1)
                const int tg = tb / 8 + 2 * h + (mi & 1), rg = 2 * jp + (mi >> 1);
                const uint32_t addr = (tg < tg8 && rg < nrv) ? vb + tg * vtg + rg * vrg + mr * 16 : zline;
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(addr, b0, b1, b2, b3);
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
    auto by_r16 = [&](int r, auto &&f) { dispatch(std::integral_constant<int, NT / 2>{}, r, f); };

    const int64_t rec_idx = is_tail      ? p.tail_rec_base + ((int)blockIdx.x - p.num_chunks)
                            : ch.nch == 1 ? (int64_t)p.num_chunks + ch.erec  // the entry record itself
                                          : (int64_t)blockIdx.x;
    float *rec = p.rec + rec_idx * recf;
    if (is_tail) {
        // tail item: query qi, KV head g, tokens [t0, t0 + ntok) of qi's dense tail
        const int item = (int)blockIdx.x - p.num_chunks, S = p.tail_splits;
        const int qi = item / (p.hkv * S), sp = item % S;
        g = (item / S) % p.hkv;
        const int64_t o0 = p.tail_offsets[qi], o1 = p.tail_offsets[qi + 1];
        const int T = (int)(o1 - o0);
        if (sp == S - 1 && T > S * kTailTokens && lane == 0) atomicCAS(p.status, 0, (int32_t)MILO_ERR_DEVICE_BOUNDS);
        const int t0 = sp * kTailTokens;
        ntok = max(0, min(t0 + kTailTokens, T) - t0);
        nrk = nrv = NT;
        // q~ = scale * log2(e) * q of the G heads of query qi, as score A fragments
#pragma unroll 1
        for (int ks = 0; ks < KD; ++ks) {
            float x[4] = {0.f, 0.f, 0.f, 0.f};
            if (r4 < p.G) {
                const uint16_t *qr = p.q + ((int64_t)qi * p.hq + g * p.G + r4) * D + 16 * ks + 2 * c4;
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
        // K then V: one box of kTailTokens rows x 8 columns per column group
        constexpr uint32_t kBox = kTailTokens * 16, kHalf = NT * kBox;
        if (ntok > 0) {
            if (lane == 0) {
                mbar_arrive_tx(bar0, 2 * kHalf);
#pragma unroll 1
                for (int c = 0; c < NT; ++c) {
                    tma_load_3d(smem_u32(smem) + c * kBox, &tmap_k, 8 * c, g, (int)(o0 + t0), bar0);
                    tma_load_3d(smem_u32(smem) + kHalf + c * kBox, &tmap_v, 8 * c, g, (int)(o0 + t0), bar0);
                }
            }
            __syncwarp();
            mbar_wait(bar0, 0, p.status);
        }
#pragma unroll 1
        for (int tb = 0; tb < ntok; tb += kTile)
            tile(std::integral_constant<int, NT / 2>{}, smem_u32(smem), 128, kBox, smem_u32(smem) + kHalf, 128, kBox,
                 tb, kTailTokens / 8, ntok);
        // the values are already in the head dimension: o = v~
        l_w = quad_sum(l_w);
#pragma unroll
        for (int n = 0; n < NT; ++n)
            __stcg(reinterpret_cast<float2 *>(rec + r4 * D + 8 * n + 2 * c4),
                   make_float2(vacc[n][0] + vacc[n][2], vacc[n][1] + vacc[n][3]));
        if (c4 == 0) {
            __stcg(rec + 8 * D + r4, ntok > 0 ? m_w : -INFINITY);
            __stcg(rec + 8 * D + 8 + r4, ntok > 0 ? l_w : 0.f);
        }
        count_record(p, g, lane);
        return;
    }

    const int np = ps.total();
    const int r16 = (max(nrk, nrv) + 1) / 2;
    // wait for piece k; afterwards release its slot and bring piece k + 2 into it
    auto wait_piece = [&](int k) {
        mbar_wait(bar0 + 8 * (k & 1), (k >> 1) & 1, p.status);
        return smem_u32(smem) + (k & 1) * kPieceBytes;
    };
    auto release_piece = [&](int k) {
        // the slot's reads are ordered before the async-proxy write
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0 && k + 2 < np) issue(k + 2);
    };
    // P^K pieces (three loops over the piece kinds keep each kind's registers
    // local to its loop)
    {
        // q rows of KV head g as the projection's B fragments (q^T)
        uint32_t qa[KD][2];
        const bool row_ok = r4 < p.rows_g;
        const uint16_t *qr = p.q + ((int64_t)(r4 / p.G) * p.hq + g * p.G + r4 % p.G) * D + 2 * c4;
#pragma unroll
        for (int ks = 0; ks < KD; ++ks) {
            qa[ks][0] = row_ok ? *reinterpret_cast<const uint32_t *>(qr + 16 * ks) : 0u;
            qa[ks][1] = row_ok ? *reinterpret_cast<const uint32_t *>(qr + 16 * ks + 8) : 0u;
        }
#pragma unroll 1
        for (int k = 0; k < ps.npk; ++k) {
            const uint32_t slot = wait_piece(k);
            // q~ for the 16-rank steps of rank groups [r0, r1): A = P^K (16 ranks x
            // 16 columns, cores (rg - r0, cg) of this piece), B = q^T, so that one
            // product covers 16 ranks; the accumulator [rank][row] is split into
            // bf16 hi + lo and transposed (movmatrix) into the score A layout.
            const int r0 = k * ps.rpp, r1 = min(r0 + ps.rpp, nrk);
            dispatch(std::integral_constant<int, L::kRanksPerPiece / 16>{}, (r1 - r0 + 1) / 2, [&](auto nkc) {
                constexpr int NK = decltype(nkc)::value;
                float acc[NK][2][4];
#pragma unroll
                for (int j = 0; j < NK; ++j)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[j][0][e] = acc[j][1][e] = 0.f;
#pragma unroll
                for (int ks = 0; ks < KD; ++ks) {
#pragma unroll
                    for (int j = 0; j < NK; ++j) {
                        // matrices: (2j, 2ks), (2j + 1, 2ks), (2j, 2ks + 1), (2j + 1, 2ks + 1)
                        const int rl = 2 * j + (mi & 1);
                        const uint32_t addr =
                            r0 + rl < r1 ? slot + (rl * NT + 2 * ks + (mi >> 1)) * 128 + mr * 16 : zline;
                        uint32_t a[4];
                        ldsm_x4(addr, a[0], a[1], a[2], a[3]);
                        mma16816(acc[j][ks & 1], a, qa[ks][0], qa[ks][1]);
                    }
                }
#pragma unroll
                for (int j = 0; j < NK; ++j) {
                    // acc: ranks 16 kk + r4 (regs 0, 1) and + 8 (regs 2, 3) for rows 2 c4, 2 c4 + 1
                    uint32_t hi0, lo0, hi1, lo1;
                    split_hi_lo((acc[j][0][0] + acc[j][1][0]) * p.scale_log2,
                                (acc[j][0][1] + acc[j][1][1]) * p.scale_log2, hi0, lo0);
                    split_hi_lo((acc[j][0][2] + acc[j][1][2]) * p.scale_log2,
                                (acc[j][0][3] + acc[j][1][3]) * p.scale_log2, hi1, lo1);
                    sq[(r0 / 2 + j) * 32 + lane] = make_uint4(movm_t(hi0), movm_t(lo0), movm_t(hi1), movm_t(lo1));
                }
            });
            __syncwarp();
            release_piece(k);
        }
    }
#pragma unroll 1
    for (int k = ps.npk; k < ps.npk + ps.nc; ++k) {
        const uint32_t slot = wait_piece(k);
        const int t0 = (k - ps.npk) * ps.tpp * kTile;
        const int nv = min(ps.tpp * kTile, ntok - t0);  // valid tokens of this piece
        const int r8 = min(t0 + ps.tpp * kTile, ch.tok8) - t0;
        const uint32_t vb = slot + (uint32_t)r8 * nrk * 16;
        by_r16(r16, [&](auto r16c) {
#pragma unroll 1
            for (int tb = 0; tb < nv; tb += kTile)
                tile(r16c, slot, nrk * 128, 128, vb, nrv * 128, 128, tb, r8 / 8, nv);
        });
        release_piece(k);
    }
    float o[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
#pragma unroll 1
    for (int k = ps.npk + ps.nc; k < np; ++k) {
        const uint32_t slot = wait_piece(k);
        // back-projection over rank 8-groups [r0, r1): 16-rank k-steps of v~
        const int r0 = (k - ps.npk - ps.nc) * ps.rpp, r1 = min(r0 + ps.rpp, nrv);
#pragma unroll
        for (int ks = 0; ks < NT / 2; ++ks) {
            if (2 * ks >= r0 && 2 * ks < r1) {
                uint32_t a[4];
                split_hi_lo(vacc[2 * ks][0] + vacc[2 * ks][2], vacc[2 * ks][1] + vacc[2 * ks][3], a[0], a[1]);
                split_hi_lo(vacc[2 * ks + 1][0] + vacc[2 * ks + 1][2], vacc[2 * ks + 1][1] + vacc[2 * ks + 1][3],
                            a[2], a[3]);
#pragma unroll
                for (int cp = 0; cp < NT / 2; ++cp) {
                    // matrices (transposed): (2ks, 2cp), (2ks + 1, 2cp), (2ks, 2cp + 1), (2ks + 1, 2cp + 1)
                    const int jg = 2 * ks + (mi & 1), cg = 2 * cp + (mi >> 1);
                    const uint32_t addr = jg < r1 ? slot + ((jg - r0) * NT + cg) * 128 + mr * 16 : zline;
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_t(addr, b0, b1, b2, b3);
                    mma16816(o[2 * cp], a, b0, b1);
                    mma16816(o[2 * cp + 1], a, b2, b3);
                }
            }
        }
        release_piece(k);
    }
    l_w = quad_sum(l_w);
#pragma unroll
    for (int n = 0; n < NT; ++n)
        __stcg(reinterpret_cast<float2 *>(rec + r4 * D + 8 * n + 2 * c4),
               make_float2(o[n][0] + o[n][2], o[n][1] + o[n][3]));
    if (c4 == 0) {
        __stcg(rec + 8 * D + r4, m_w);
        __stcg(rec + 8 * D + 8 + r4, l_w);
    }
    if (ch.nch > 1) {
        // the entry's last chunk to finish merges its chunk records
        __threadfence();
        __syncwarp();
        uint32_t old = 0;
        if (lane == 0) old = atomicAdd(&p.entry_cnt[ch.erec], 1u);
        old = __shfl_sync(0xffffffffu, old, 0);
        if (old != (uint32_t)ch.nch - 1) return;
        if (lane == 0) p.entry_cnt[ch.erec] = 0u;  // ready for the next call
        __threadfence();
        merge_entry<D>(p, ch.c0, ch.nch, p.rec + ((int64_t)p.num_chunks + ch.erec) * recf, lane);
    }
    count_record(p, g, lane);
}

}  // namespace

cudaError_t launch_chunks(const DecodeParams &p, const void *tmap_k, const void *tmap_v, cudaStream_t stream)
{
    const CUtensorMap &mk = *static_cast<const CUtensorMap *>(tmap_k);
    const CUtensorMap &mv = *static_cast<const CUtensorMap *>(tmap_v);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.num_chunks + (p.has_tail ? p.num_tail_items : 0) + p.hkv * kMergeWarpsPerHead);
    cfg.blockDim = dim3(32);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    static int configured[2] = {0, 0};
    const int w = p.d == 64 ? 0 : 1;
    const void *fn = w == 0 ? reinterpret_cast<const void *>(chunk_kernel<64>)
                            : reinterpret_cast<const void *>(chunk_kernel<128>);
    const int smem = w == 0 ? CLay<64>::kTotal : CLay<128>::kTotal;
    if (!configured[w]) {
        cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        // several thread blocks per SM need the largest shared-memory carveout
        e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        if (e != cudaSuccess) return e;
        configured[w] = 1;
    }
    cfg.dynamicSmemBytes = (size_t)smem;
    return w == 0 ? cudaLaunchKernelEx(&cfg, chunk_kernel<64>, p, mk, mv)
                  : cudaLaunchKernelEx(&cfg, chunk_kernel<128>, p, mk, mv);
}

}  // namespace milo
