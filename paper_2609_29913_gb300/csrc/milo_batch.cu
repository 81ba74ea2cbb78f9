// milo_batch.cu -- the prefix part of a decode call with many query rows per
// KV head (batched decode over one shared prefix), on the fifth-generation
// tensor cores: tcgen05.mma with fp32 accumulators in tensor memory.
//
// For a KV head g the call has R = batch x G query rows.  They are cut into
// tiles of 128 rows, the M side of every product, so each product serves 128
// rows at once (Eq. 3 substituted into Eq. 1, Alg. 1 Stage 2):
//
//   projection       Q~  = Q P^K^T       A = q rows (K = d),      B = P^K  (N = ranks)
//   scores           S   = Q~ C^K^T      A = q~ hi, lo (K = ranks), B = C^K tile (N = 64 tokens)
//   values           V~ += P C^V         A = p hi, lo (K = tokens), B = C^V tile (N = ranks)
//   back-projection  O  += V~ P^V        A = v~ hi, lo (K = ranks), B = P^V  (N = d)
//
// q~, p and v~ are fp32 values that enter a product as two bf16 operands,
// the value rounded to bf16 ("hi") and its rounding residual ("lo"), so they
// keep ~16 significant bits; the factors and q are bf16 data and enter once.
// Scores are in log2 units: q~ carries softmax scale x log2(e).
//
// Work: the prefix (every entry's tokens, KV-head-major, then table order)
// is cut on the host into near-equal shares at 32-token boundaries
// (segments); one thread block per (share, row tile) walks its share's
// segments in order.  Consecutive segments of one KV head form a run: its
// softmax state (m, l) and its output O stay in the block across segments
// (O accumulates every segment's back-projection in tensor memory), and the
// run adds its result into the plan's per-row accumulators once, at its end
// (the shared-reference merge of milo_merge.cuh), or lists it as records.
//
// A block of 192 threads, one per SM (224 KB of shared memory, all 512
// tensor-memory columns):
//   warp 0, lane 0   producer: bulk copies of the segment pieces (P^K, then
//                    C^K + C^V rows of whole 64-token tiles up to 32 KB,
//                    then P^V) into a ring of two 32 KB slots;
//   warp 1           owns the tensor memory; lane 0 issues every MMA;
//   warps 2-5        softmax: thread t owns row t of the tile and tensor
//                    memory lane t (warp w reaches lanes 32 (w % 4) ..).
// Within a segment the score tile j + 1 is computed while the softmax works
// on tile j (two score buffers in tensor memory, two p buffers in shared
// memory).  The online softmax raises a row's reference maximum lazily (only
// when a score passes it by kLazyTc), rescaling V~ and O in tensor memory
// when it does.
//
// Every mbarrier wait is bounded (~2 s): a wait that gives up sets
// MILO_ERR_TIMEOUT in the status word and a shared abort flag, after which
// every role skips its remaining work, so the block always ends.
#include <cuda.h>
#include <cuda_bf16.h>

#include "milo.h"
#include "milo_internal.h"
#include "milo_merge.cuh"
#include "milo_ptx.cuh"

namespace milo {
namespace {

constexpr int kTcThreads = 192;
constexpr int kTcSlots = 2;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;    // two score tiles of kTcTok columns
constexpr uint32_t kColQ = 128;  // projection result q~ (fp32, up to 128 ranks)
constexpr uint32_t kColV = 256;  // rank-space values v~ (fp32, up to 128 ranks)
constexpr uint32_t kColO = 384;  // output O (fp32, d columns)
constexpr float kLazyTc = 8.f;   // a row's reference maximum moves when a score passes it by this

// mbarriers; (n) = arrivals per phase
enum : int {
    TB_FULL = 0,                    // [kTcSlots] piece landed (1 + bytes)
    TB_EMPTY = TB_FULL + kTcSlots,  // [kTcSlots] MMAs reading the piece done (commit)
    TB_QROWS = TB_EMPTY + kTcSlots, // q rows of a run staged (4 softmax warps)
    TB_PROJ,                        // projection done (commit)
    TB_QT,                          // q~ staged (4)
    TB_SFULL,                       // [2] score tile done (commit)
    TB_SFREE = TB_SFULL + 2,        // [2] score tile read (4)
    TB_PREADY = TB_SFREE + 2,       // [2] p tile staged (4)
    TB_PVDONE = TB_PREADY + 2,      // [2] value products of that p tile done (commit)
    TB_VDONE = TB_PVDONE + 2,       // every value product of a segment done (commit)
    TB_VSTAGED,                     // v~ staged for the back-projection (4)
    TB_BPDONE,                      // back-projection done (commit)
    TB_FIN,                         // every MMA of the block done (commit)
    TB_NBAR
};

template <int D>
struct TcLay {
    static constexpr int kQ = kTcSlots * kTcSlot;                 // after the ring: q rows, cores [16 row groups][D/8]
    static constexpr int kQt = kQ + kTcRows * D * 2;              // q~ hi, then lo: cores [16][D/8] each
    static constexpr int kQtHalf = kTcRows * D * 2;
    static constexpr int kP = kQt + 2 * kQtHalf;                  // two p tiles (hi, lo: cores [16][8] each);
    static constexpr int kPHalf = kTcRows * kTcTok * 2;           //   v~ hi, lo at a segment's end
    static constexpr int kPBuf = 2 * kPHalf;
    static constexpr int kBar = kP + 2 * kPBuf;
    static constexpr int kFlag = kBar + TB_NBAR * 8;              // abort flag, tensor-memory base
    static constexpr int kTotal = kFlag + 16;
    static_assert(2 * kQtHalf <= 2 * kPBuf, "v~ hi and lo fit the two p tiles");
    static_assert(kTotal <= 232448, "one block per SM");
};

// ------------------------------------------------------------ tcgen05 ----
namespace tc {
// Shared-memory matrix descriptor, no swizzle, 8x8-element cores of 16-byte
// rows: LBO = byte stride between cores along K, SBO = along M (or N).
__device__ __forceinline__ uint64_t sdesc(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | ((uint64_t)1 << 46);
}
// Instruction descriptor: M = 128, N = n, bf16 x bf16 -> f32; a_mn / b_mn:
// operand stored M- / N-major (else K-major).
__device__ __forceinline__ uint32_t idesc(bool a_mn, bool b_mn, int n)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
           ((uint32_t)(n >> 3) << 17) | ((128u >> 4) << 24);
}
__device__ __forceinline__ void umma(uint32_t d, uint64_t a, uint64_t b, uint32_t id, bool acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(id), "r"((int)acc));
}
// n products into one accumulator: step k reads A at a + k a_step and B at
// b + k b_step (bytes; the address is the descriptor's low field, in 16-byte
// units); step 0 overwrites D unless acc0.
__device__ __forceinline__ void umma_n(uint32_t d, uint64_t a, uint64_t b, uint32_t a_step, uint32_t b_step, int n,
                                       uint32_t id, bool acc0)
{
#pragma unroll 1
    for (int k = 0; k < n; ++k) {
        umma(d, a, b, id, k > 0 || acc0);
        a += a_step >> 4;
        b += b_step >> 4;
    }
}
// mbarrier arrival once every MMA issued so far by this thread has completed
__device__ __forceinline__ void commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
// 16 consecutive fp32 columns of this warp's 32 lanes (no wait)
__device__ __forceinline__ void ld16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void st16(uint32_t taddr, const float (&v)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
        "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
        "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])),
        "r"(__float_as_uint(v[11])), "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])),
        "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15]))
        : "memory");
}
__device__ __forceinline__ void wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
}  // namespace tc

// 16 fp32 values of one row as bf16 hi + lo into two K-major cores each
// (columns 8c .. 8c + 15 of the row): hi cores at `hi`, hi + 128, lo cores at
// `lo`, lo + 128 (each address already at the row's 16-byte line).
__device__ __forceinline__ void put16(uint8_t *hi, uint8_t *lo, const float (&x)[16])
{
    uint32_t h[8], l[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) split_hi_lo(x[2 * j], x[2 * j + 1], h[j], l[j]);
    *reinterpret_cast<uint4 *>(hi) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4 *>(hi + 128) = make_uint4(h[4], h[5], h[6], h[7]);
    *reinterpret_cast<uint4 *>(lo) = make_uint4(l[0], l[1], l[2], l[3]);
    *reinterpret_cast<uint4 *>(lo + 128) = make_uint4(l[4], l[5], l[6], l[7]);
}

// Bounded wait that also gives up once another thread of the block has
// (the shared abort flag); false when it gave up.
__device__ __forceinline__ bool tc_wait(uint32_t bar, uint32_t parity, int32_t *status, volatile int *abort_flag)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 32; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer() - t0 > kTimeoutNs) {
            atomicCAS(status, 0, (int32_t)MILO_ERR_TIMEOUT);
            *abort_flag = 1;
            return false;
        }
    }
}

// What a segment (tokens [t0, t1) of one entry) needs, as both the producer
// and the MMA issuer walk it.
struct SegPlan {
    int64_t ck, pk, cv, pv;  // packed byte offsets (C at token 0 of the entry)
    int n8;                  // entry tokens rounded up to 8
    int rk, rv, rk8, rv8;    // ranks and rank 8-groups
    int g, t0, t1;
    int ntiles, tpp, nc;     // 64-token tiles, tiles per C piece, C pieces
    bool first_of_run, last_of_run;
    int slot;                // run record slot
};

__device__ __forceinline__ SegPlan seg_plan(const DecodeParams &p, int s)
{
    const SegDev sd = p.tc_segs[s];
    const EntryDev e = p.entries[sd.entry];
    SegPlan q;
    q.ck = e.off_ck;
    q.pk = e.off_pk;
    q.cv = e.off_cv;
    q.pv = e.off_pv;
    q.n8 = (e.n + 7) & ~7;
    q.rk = e.rk;
    q.rv = e.rv;
    q.rk8 = (e.rk + 7) / 8;
    q.rv8 = (e.rv + 7) / 8;
    q.g = e.g;
    q.t0 = sd.t0;
    q.t1 = sd.t1;
    q.ntiles = (sd.t1 - sd.t0 + kTcTok - 1) / kTcTok;
    const int row_bytes = kTcTok * (q.rk8 + q.rv8) * 16;  // one tile's C^K + C^V
    q.tpp = row_bytes > 0 ? max(1, kTcSlot / row_bytes) : q.ntiles;
    q.nc = row_bytes > 0 ? (q.ntiles + q.tpp - 1) / q.tpp : 0;
    q.first_of_run = (sd.flags & kSegFirstOfRun) != 0;
    q.last_of_run = (sd.flags & kSegLastOfRun) != 0;
    q.slot = sd.slot;
    return q;
}

// Rows of C piece c of a segment: tokens [a, a + rows) of the entry, rows a
// multiple of 8 (the piece's tiles, the last one cut at the segment end and
// rounded up to 8 within the entry).
__device__ __forceinline__ void c_piece_rows(const SegPlan &q, int c, int &a, int &rows)
{
    a = q.t0 + c * q.tpp * kTcTok;
    const int b = min(q.t0 + (c + 1) * q.tpp * kTcTok, q.t1);
    rows = min((b + 7) & ~7, q.n8) - a;
}

template <int D>
__global__ void __launch_bounds__(kTcThreads, 1) batch_tc_kernel(const __grid_constant__ DecodeParams p)
{
    using L = TcLay<D>;
    constexpr int DG = D / 8;  // 8-column groups of the head dimension (also rank groups of a full rank)
    extern __shared__ __align__(128) uint8_t smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t sbase = smem_u32(smem);
    const uint32_t bar0 = smem_u32(smem + L::kBar);
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::kFlag);
    const int share = (int)blockIdx.x / p.tc_ntile, tile = (int)blockIdx.x % p.tc_ntile;
    const int s_begin = p.tc_cta_begin[share], s_end = p.tc_cta_begin[share + 1];

    pdl_trigger();
    // zero the ring, q rows, q~ and p areas: every later read past a piece's
    // data (rank and token padding of the products) sees finite values
    for (int i = tid; i < L::kBar / 16; i += kTcThreads) reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
    if (tid == 0) {
        for (int i = 0; i < kTcSlots; ++i) {
            mbar_init(bar(TB_FULL + i), 1);
            mbar_init(bar(TB_EMPTY + i), 1);
        }
        mbar_init(bar(TB_QROWS), 4);
        mbar_init(bar(TB_PROJ), 1);
        mbar_init(bar(TB_QT), 4);
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(TB_SFULL + i), 1);
            mbar_init(bar(TB_SFREE + i), 4);
            mbar_init(bar(TB_PREADY + i), 4);
            mbar_init(bar(TB_PVDONE + i), 1);
        }
        mbar_init(bar(TB_VDONE), 1);
        mbar_init(bar(TB_VSTAGED), 4);
        mbar_init(bar(TB_BPDONE), 1);
        mbar_init(bar(TB_FIN), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    tc::fence_proxy();
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(smem + L::kFlag + 8)),
                     "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(smem + L::kFlag + 8);

    if (warp == 0) {
        // ------------------------------------------------ producer
        // The packed arena and the plan's segment list belong to the plan,
        // which no kernel writes: the pieces may stream before the wait on
        // the preceding grid.
        if (lane == 0) {
            int n = 0;  // pieces issued
            auto issue = [&](auto &&copies) -> bool {
                const int sl = n % kTcSlots;
                if (n >= kTcSlots && !tc_wait(bar(TB_EMPTY + sl), ((n / kTcSlots) - 1) & 1, p.status, abort_flag))
                    return false;
                copies(sbase + (uint32_t)sl * kTcSlot, bar(TB_FULL + sl));
                ++n;
                return true;
            };
            bool ok = true;
            for (int s = s_begin; ok && s < s_end; ++s) {
                const SegPlan q = seg_plan(p, s);
                if (q.rk > 0)
                    ok = issue([&](uint32_t dst, uint32_t b) {
                        const uint32_t bytes = (uint32_t)q.rk8 * D * 16;
                        mbar_arrive_tx(b, bytes);
                        bulk_g2s(dst, p.packed + q.pk, bytes, b);
                    });
                for (int c = 0; ok && c < q.nc; ++c)
                    ok = issue([&](uint32_t dst, uint32_t b) {
                        int a, rows;
                        c_piece_rows(q, c, a, rows);
                        const uint32_t kb = (uint32_t)rows * q.rk8 * 16, vb = (uint32_t)rows * q.rv8 * 16;
                        mbar_arrive_tx(b, kb + vb);
                        if (kb) bulk_g2s(dst, p.packed + q.ck + (int64_t)a * q.rk8 * 16, kb, b);
                        if (vb) bulk_g2s(dst + kb, p.packed + q.cv + (int64_t)a * q.rv8 * 16, vb, b);
                    });
                if (ok && q.rv > 0)
                    ok = issue([&](uint32_t dst, uint32_t b) {
                        const uint32_t bytes = (uint32_t)q.rv8 * D * 16;
                        mbar_arrive_tx(b, bytes);
                        bulk_g2s(dst, p.packed + q.pv, bytes, b);
                    });
            }
            // the block may not end with copies into its shared memory in
            // flight: wait (bounded) for the last pieces to land
            for (int k = max(0, n - kTcSlots); k < n; ++k)
                mbar_wait(bar(TB_FULL + k % kTcSlots), (k / kTcSlots) & 1, p.status);
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        pdl_wait();
        if (lane == 0) {
            int n = 0;      // pieces consumed (in producer order)
            int J = 0;      // score tiles issued (global over segments)
            int kseg = 0;   // segments
            int krun = 0;   // runs
            bool o_acc = false;
            bool ok = true;
            auto take = [&](int &slot) {
                slot = n % kTcSlots;
                ok = ok && tc_wait(bar(TB_FULL + slot), (n / kTcSlots) & 1, p.status, abort_flag);
                ++n;
                tc::fence_after();
                return sbase + (uint32_t)slot * kTcSlot;
            };
            const uint32_t q_u = sbase + L::kQ, qt_u = sbase + L::kQt, p_u = sbase + L::kP;
            for (int s = s_begin; ok && s < s_end; ++s) {
                const SegPlan q = seg_plan(p, s);
                const int nk16 = (q.rk8 + 1) / 2, nv16 = (q.rv8 + 1) / 2;  // 16-rank steps
                if (q.first_of_run) {
                    ok = ok && tc_wait(bar(TB_QROWS), krun & 1, p.status, abort_flag);
                    ++krun;
                    o_acc = false;
                    tc::fence_after();
                }
                // projection q~ = Q P^K^T into kColQ (N = 16 nk16 ranks, K = d)
                if (q.rk > 0) {
                    int sl;
                    const uint32_t pk = take(sl);
                    if (ok)
                        tc::umma_n(tmem + kColQ, tc::sdesc(q_u, 128, DG * 128), tc::sdesc(pk, 128, DG * 128), 256, 256,
                                   D / 16, tc::idesc(false, false, 16 * nk16), false);
                    tc::commit(bar(TB_EMPTY + sl));
                }
                tc::commit(bar(TB_PROJ));
                ok = ok && tc_wait(bar(TB_QT), kseg & 1, p.status, abort_flag);
                tc::fence_after();
                // tiles: S_j is issued before the value products of tile j - 1
                int cur_slot = -1, prev_slot = -1;
                uint32_t cur = 0, cvb = 0, prev_cvb = 0;
                const int J0 = J;
                for (int j = 0; ok && j <= q.ntiles; ++j) {
                    if (j < q.ntiles) {
                        const int c = q.nc > 0 ? j / q.tpp : 0, jj = q.nc > 0 ? j % q.tpp : 0;
                        if (q.nc > 0 && jj == 0) {
                            prev_slot = cur_slot;
                            prev_cvb = cvb;
                            cur = take(cur_slot);
                            int a, rows;
                            c_piece_rows(q, c, a, rows);
                            cvb = cur + (uint32_t)rows * q.rk8 * 16;
                        }
                        const int b = (J0 + j) & 1, u = (J0 + j) >> 1;
                        if (J0 + j >= 2) ok = ok && tc_wait(bar(TB_SFREE + b), (u - 1) & 1, p.status, abort_flag);
                        tc::fence_after();
                        if (ok && q.rk > 0) {
                            const uint32_t kt = cur + (uint32_t)jj * 8 * q.rk8 * 128;
                            const uint32_t id = tc::idesc(false, false, kTcTok);
                            tc::umma_n(tmem + kColS + kTcTok * b, tc::sdesc(qt_u, 128, DG * 128),
                                       tc::sdesc(kt, 128, q.rk8 * 128), 256, 256, nk16, id, false);
                            tc::umma_n(tmem + kColS + kTcTok * b, tc::sdesc(qt_u + L::kQtHalf, 128, DG * 128),
                                       tc::sdesc(kt, 128, q.rk8 * 128), 256, 256, nk16, id, true);
                        }
                        tc::commit(bar(TB_SFULL + b));
                    }
                    if (j > 0) {
                        // value products of tile jt = j - 1
                        const int jt = j - 1, Jt = J0 + jt, b = Jt & 1;
                        const int jj = q.nc > 0 ? jt % q.tpp : 0;
                        // the tile's piece: the current one, unless tile j opened a new piece
                        const bool in_prev = q.nc > 0 && j < q.ntiles && (j % q.tpp) == 0;
                        const uint32_t vbase = in_prev ? prev_cvb : cvb;
                        ok = ok && tc_wait(bar(TB_PREADY + b), (Jt >> 1) & 1, p.status, abort_flag);
                        tc::fence_after();
                        if (ok && q.rv > 0) {
                            const uint32_t vt = vbase + (uint32_t)jj * 8 * q.rv8 * 128;
                            const uint32_t id = tc::idesc(false, true, 16 * nv16);
                            const uint32_t pa = p_u + (uint32_t)b * L::kPBuf;
                            tc::umma_n(tmem + kColV, tc::sdesc(pa, 128, 8 * 128), tc::sdesc(vt, q.rv8 * 128, 128), 256,
                                       2 * q.rv8 * 128, kTcTok / 16, id, jt > 0);
                            tc::umma_n(tmem + kColV, tc::sdesc(pa + L::kPHalf, 128, 8 * 128),
                                       tc::sdesc(vt, q.rv8 * 128, 128), 256, 2 * q.rv8 * 128, kTcTok / 16, id, true);
                        }
                        tc::commit(bar(TB_PVDONE + b));
                        // the last tile of a piece releases its slot
                        if (q.nc > 0 && (jt % q.tpp == q.tpp - 1 || jt == q.ntiles - 1))
                            tc::commit(bar(TB_EMPTY + (in_prev ? prev_slot : cur_slot)));
                    }
                }
                J = J0 + q.ntiles;
                tc::commit(bar(TB_VDONE));
                // back-projection O += V~ P^V (N = d, K = 16 nv16 ranks)
                int pv_slot = -1;
                uint32_t pvu = 0;
                if (q.rv > 0) pvu = take(pv_slot);
                ok = ok && tc_wait(bar(TB_VSTAGED), kseg & 1, p.status, abort_flag);
                tc::fence_after();
                if (ok && q.rv > 0) {
                    const uint32_t id = tc::idesc(false, true, D);
                    tc::umma_n(tmem + kColO, tc::sdesc(p_u, 128, DG * 128), tc::sdesc(pvu, DG * 128, 128), 256,
                               2 * DG * 128, nv16, id, o_acc);
                    tc::umma_n(tmem + kColO, tc::sdesc(p_u + L::kQtHalf, 128, DG * 128), tc::sdesc(pvu, DG * 128, 128),
                               256, 2 * DG * 128, nv16, id, true);
                    o_acc = true;
                }
                tc::commit(bar(TB_BPDONE));
                if (q.rv > 0) tc::commit(bar(TB_EMPTY + pv_slot));
                ++kseg;
            }
            tc::commit(bar(TB_FIN));
            mbar_wait(bar(TB_FIN), 0, p.status);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ softmax
        const int quad = warp & 3;                // tensor-memory lane quarter of this warp
        const int rl = 32 * quad + lane;          // row within the tile
        const int row = tile * kTcRows + rl;      // the KV head's query row (batch x heads)
        const bool row_ok = row < p.rows_g;
        const uint32_t tl = tmem + ((uint32_t)(32 * quad) << 16);
        uint8_t *q_s = smem + L::kQ, *qt_s = smem + L::kQt, *p_s = smem + L::kP;
        const int rg8 = rl >> 3, r8 = rl & 7;     // core row group and row within the core
        pdl_wait();  // q and the accumulators belong to the preceding grids until here
        int J = 0, kseg = 0;
        bool ok = true;
        float m = -INFINITY, l = 0.f;
        bool o_written = false, first_tile = true;
        uint32_t ref = 0u;
        auto arrive = [&](int b) {
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(b));
        };
        // the warp-collective tensor-memory accesses after a wait need every
        // lane to agree on its outcome
        auto wwait = [&](int b, int parity) {
            ok = __all_sync(0xffffffffu, ok && tc_wait(bar(b), (uint32_t)parity & 1u, p.status, abort_flag));
        };
        for (int s = s_begin; s < s_end; ++s) {
            const SegPlan q = seg_plan(p, s);
            const int g = q.g;
            if (q.first_of_run) {
                // this run's q rows as the projection's A operand
                const uint4 *qr = reinterpret_cast<const uint4 *>(
                    p.q + ((int64_t)(row / p.G) * p.hq + g * p.G + row % p.G) * D);
#pragma unroll 4
                for (int c = 0; c < DG; ++c) {
                    const uint4 v = row_ok ? __ldcg(qr + c) : make_uint4(0u, 0u, 0u, 0u);
                    *reinterpret_cast<uint4 *>(q_s + (rg8 * DG + c) * 128 + r8 * 16) = v;
                }
                tc::fence_proxy();
                arrive(TB_QROWS);
                m = -INFINITY;
                l = 0.f;
                o_written = false;
                first_tile = true;
            }
            // q~ = scale log2(e) Q P^K^T as hi and lo A operands (rank groups
            // past the rank: zero)
            wwait(TB_PROJ, kseg);
            tc::fence_after();
            const int nk16 = (q.rk8 + 1) / 2, nv16 = (q.rv8 + 1) / 2;
            if (ok) {
#pragma unroll 1
                for (int c = 0; c < nk16; ++c) {
                    float v[16];
                    tc::ld16(tl + kColQ + 16 * c, v);
                    tc::wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[i] = 16 * c + i < q.rk ? v[i] * p.scale_log2 : 0.f;
                    uint8_t *hi = qt_s + (rg8 * DG + 2 * c) * 128 + r8 * 16;
                    put16(hi, hi + L::kQtHalf, v);
                }
            }
            tc::fence_proxy();
            tc::fence_before();
            arrive(TB_QT);
            // tiles
            const int ntok = q.t1 - q.t0;
#pragma unroll 1
            for (int j = 0; j < q.ntiles; ++j, ++J) {
                const int b = J & 1;
                wwait(TB_SFULL + b, J >> 1);
                tc::fence_after();
                float sv[kTcTok];
                if (ok && q.rk > 0) {
#pragma unroll
                    for (int c = 0; c < kTcTok / 16; ++c) {
                        float v[16];
                        tc::ld16(tl + kColS + kTcTok * b + 16 * c, v);
#pragma unroll
                        for (int i = 0; i < 16; ++i) sv[16 * c + i] = v[i];
                    }
                    tc::wait_ld();
                } else {
#pragma unroll
                    for (int i = 0; i < kTcTok; ++i) sv[i] = 0.f;
                }
                tc::fence_before();
                arrive(TB_SFREE + b);
                const int nvalid = min(kTcTok, ntok - kTcTok * j);
                float mx = -INFINITY;
#pragma unroll
                for (int i = 0; i < kTcTok; ++i) {
                    sv[i] = i < nvalid ? sv[i] : -INFINITY;
                    mx = fmaxf(mx, sv[i]);
                }
                // lazy rescale: the reference moves only when a score passes it
                // by kLazyTc; V~ and O, already summed against the old one,
                // are multiplied by 2^(m_old - m_new) in tensor memory
                const bool need = mx > m + kLazyTc;
                if (__any_sync(0xffffffffu, need)) {
                    const float mn = need ? mx : m;
                    const float alpha = need ? exp2_diff(m, mn) : 1.f;
                    if (j > 0) {
                        // the value products of tile j - 1 (and every earlier
                        // product) must be done
                        const int Jp = J - 1;
                        wwait(TB_PVDONE + (Jp & 1), Jp >> 1);
                        tc::fence_after();
                        if (ok && q.rv > 0) {
#pragma unroll 1
                            for (int c = 0; c < nv16; ++c) {
                                float v[16];
                                tc::ld16(tl + kColV + 16 * c, v);
                                tc::wait_ld();
#pragma unroll
                                for (int i = 0; i < 16; ++i) v[i] *= alpha;
                                tc::st16(tl + kColV + 16 * c, v);
                            }
                        }
                    }
                    if (ok && o_written) {
#pragma unroll 1
                        for (int c = 0; c < D / 16; ++c) {
                            float v[16];
                            tc::ld16(tl + kColO + 16 * c, v);
                            tc::wait_ld();
#pragma unroll
                            for (int i = 0; i < 16; ++i) v[i] *= alpha;
                            tc::st16(tl + kColO + 16 * c, v);
                        }
                    }
                    tc::wait_st();
                    tc::fence_before();
                    l *= alpha;
                    m = mn;
                }
                if (first_tile) {
                    ref = publish_ref(p, g, row, row_ok, 0, m);
                    first_tile = false;
                }
                float pr[kTcTok];
                float ls = 0.f;
#pragma unroll
                for (int i = 0; i < kTcTok; ++i) {
                    pr[i] = ex2_approx(sv[i] - m);  // a masked score gives 0
                    ls += pr[i];
                }
                l += ls;
                // p tile b is free once the value products of tile J - 2 are done
                if (j >= 2) {
                    wwait(TB_PVDONE + b, (J - 2) >> 1);
                    tc::fence_after();
                }
                uint8_t *pb = p_s + b * L::kPBuf + (rg8 * (kTcTok / 8)) * 128 + r8 * 16;
#pragma unroll
                for (int h = 0; h < kTcTok / 16; ++h) {
                    float x[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) x[i] = pr[16 * h + i];
                    put16(pb + 2 * h * 128, pb + L::kPHalf + 2 * h * 128, x);
                }
                tc::fence_proxy();
                arrive(TB_PREADY + b);
            }
            // segment end: V~ as the back-projection's hi and lo A operands
            // (in the p tiles, free once every value product is done)
            wwait(TB_VDONE, kseg);
            tc::fence_after();
            if (ok && q.rv > 0) {
#pragma unroll 1
                for (int c = 0; c < nv16; ++c) {
                    float v[16];
                    tc::ld16(tl + kColV + 16 * c, v);
                    tc::wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[i] = 16 * c + i < q.rv ? v[i] : 0.f;
                    uint8_t *hi = p_s + (rg8 * DG + 2 * c) * 128 + r8 * 16;
                    put16(hi, hi + L::kQtHalf, v);
                }
            }
            tc::fence_proxy();
            tc::fence_before();
            arrive(TB_VSTAGED);
            wwait(TB_BPDONE, kseg);
            tc::fence_after();
            if (q.rv > 0) o_written = true;
            ++kseg;
            if (q.last_of_run && ok) {
                // ---- the run's result into the accumulators of KV head g
                // (or, for a row group with an outlier maximum, as a record)
                const float Mref = ref ? ref_dec(ref) : m;
                const bool outlier = row_ok && m - Mref > kDirectMax;
                const uint32_t votes = __ballot_sync(0xffffffffu, outlier);
                const bool direct = ((votes >> (lane & ~7)) & 0xffu) == 0u;
                const int rgg = row >> 3;
                const int64_t rec_idx = (int64_t)q.slot * p.nrg + rgg;
                float *rec = p.rec + rec_idx * (8 * D + kRecFloatsExtra);
                const float f = row_ok && direct ? ex2_approx(m - Mref) : 0.f;
                float *arow = p.acc_o + ((int64_t)g * p.rows_max + row) * D;
#pragma unroll 1
                for (int c = 0; c < D / 16; ++c) {
                    float o[16];
                    if (o_written) {
                        tc::ld16(tl + kColO + 16 * c, o);
                        tc::wait_ld();
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) o[i] = 0.f;
                    }
                    if (!row_ok) continue;
                    if (direct) {
#pragma unroll
                        for (int i = 0; i < 16; i += 4)
                            atomicAdd(reinterpret_cast<float4 *>(arow + 16 * c + i),
                                      make_float4(f * o[i], f * o[i + 1], f * o[i + 2], f * o[i + 3]));
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; i += 4)
                            __stcg(reinterpret_cast<float4 *>(rec + r8 * D + 16 * c + i),
                                   make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]));
                    }
                }
                if (row_ok) {
                    if (direct) {
                        atomicAdd(p.acc_l + (int64_t)g * p.rows_max + row, f * l);
                    } else {
                        __stcg(rec + 8 * D + r8, m);
                        __stcg(rec + 8 * D + 8 + r8, l);
                    }
                }
                // one lane per row group lists an outlier record
                if (!direct && r8 == 0 && row_ok) {
                    const int gr = g * p.nrg + rgg;
                    const uint32_t k = atomicAdd(p.ovf_cnt + gr, 1u);
                    __stcg(reinterpret_cast<int4 *>(p.ovf_list) + (int64_t)gr * p.list_cap + k,
                           make_int4((int)rec_idx, 8 * rgg, min(8, p.rows_g - 8 * rgg), 0));
                }
                tc::fence_before();
            }
        }
    }
    // every MMA is done (the issuer waited for them) and every tensor-memory
    // read has completed: release the tensor memory
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

}  // namespace

int batch_tc_smem_bytes(int head_dim) { return head_dim == 64 ? TcLay<64>::kTotal : TcLay<128>::kTotal; }

cudaError_t launch_batch_tc(const DecodeParams &p, cudaStream_t stream)
{
    static bool configured[kMaxDevices][2] = {};
    const int which = p.d == 64 ? 0 : 1;
    const int dev = attribute_slot();
    if (dev < 0 || !configured[dev][which]) {
        cudaError_t e = which == 0 ? cudaFuncSetAttribute(batch_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                          TcLay<64>::kTotal)
                                   : cudaFuncSetAttribute(batch_tc_kernel<128>,
                                                          cudaFuncAttributeMaxDynamicSharedMemorySize, TcLay<128>::kTotal);
        if (e != cudaSuccess) return e;
        if (dev >= 0) configured[dev][which] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.tc_nshare * p.tc_ntile);
    cfg.blockDim = dim3(kTcThreads);
    cfg.dynamicSmemBytes = (size_t)batch_tc_smem_bytes(p.d);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return which == 0 ? cudaLaunchKernelEx(&cfg, batch_tc_kernel<64>, p) : cudaLaunchKernelEx(&cfg, batch_tc_kernel<128>, p);
}

}  // namespace milo
