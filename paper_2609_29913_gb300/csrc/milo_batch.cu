// milo_batch.cu -- the prefix part of a decode call with many query rows per
// KV head (batched decode over one shared prefix), on the fifth-generation
// tensor cores: tcgen05.mma with fp32 accumulators in tensor memory.
//
// For a KV head g the call has R = batch x G query rows.  They are cut into
// tiles of 128 rows, the M side of every product, so each product serves 128
// rows at once (Eq. 3 substituted into Eq. 1, Alg. 1 Stage 2):
//
//   projection       Q~  = Q P^K^T    A = q rows (smem, K = d)          B = P^K      (N = ranks)
//   scores           S   = Q~ C^K^T   A = q~ hi, lo (smem, K = ranks)   B = C^K tile (N = 64 tokens)
//   values           V~ += P C^V      A = p hi, lo (tmem, K = tokens)   B = C^V tile (N = ranks)
//   back-projection  O  += V~ P^V     A = v~ hi, lo (tmem, K = ranks)   B = P^V      (N = d)
//
// q~, p and v~ are fp32 values that enter a product as two bf16 operands,
// the value truncated to bf16 ("hi") and its residual ("lo"), so they keep
// ~15 significant bits; the factors and q are bf16 data and enter once.  Scores
// are in log2 units: q~ carries softmax scale x log2(e).
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
// A block of 320 threads, one per SM (227 KB of shared memory, all 512
// tensor-memory columns):
//   warp 0, lane 0   producer: bulk copies of the segment pieces (P^K, then
//                    C^K + C^V rows of whole 64-token tiles up to 32 KB,
//                    then P^V) into a ring of four 32 KB slots;
//   warp 1           owns the tensor memory and walks the MMA schedule as a
//                    converged warp; one elected lane issues every MMA;
//   warps 2-9        softmax, two warps per tensor-memory lane quarter (warp
//                    w reaches lanes 32 (w % 4) ..): lane t of a pair owns
//                    row t of the quarter; the pair splits every tile's
//                    columns.
// Tensor memory: two score tiles (each overwritten in place by its p hi, lo
// once read), q~ as projected, v~ (converted in place to its hi, lo at a
// segment's end), O.  The score products run two tiles ahead of the value
// products, so the softmax of tile j overlaps the products of tiles j - 1
// and j + 1.  tcgen05.mma operations of one thread execute in issue order,
// which orders a score product after the value product that read the p
// tile it overwrites, and a segment's first value product after the
// previous segment's back-projection.  At a segment's end the next
// segment's projection, q~ and first score products go ahead of this
// segment's back-projection.
//
// The online softmax raises a row's reference maximum lazily (only when a
// score passes it by kLazyTc), rescaling V~ and O in tensor memory when it
// does.  Every mbarrier wait is bounded (~2 s): a wait that gives up sets
// MILO_ERR_TIMEOUT in the status word and a shared abort flag, after which
// every role skips its remaining work, so the block always ends.
#include <cuda.h>
#include <cuda_bf16.h>

#include <type_traits>

#include "milo.h"
#include "milo_internal.h"
#include "milo_merge.cuh"
#include "milo_ptx.cuh"

namespace milo {
namespace {

constexpr int kTcThreads = 320;   // producer warp, MMA warp, 8 softmax warps
constexpr int kTcSlots = 4;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;    // two score tiles of kTcTok columns (then p hi | p lo)
constexpr uint32_t kColQ = 128;  // projection result q~ (fp32, up to 128 ranks)
constexpr uint32_t kColV = 256;  // rank-space values v~ (fp32; then v~ hi at +0, lo at +64)
constexpr uint32_t kColO = 384;  // output O (fp32, d columns)
constexpr float kLazyTc = 8.f;   // a row's reference maximum moves when a score passes it by this

// mbarriers; (n) = arrivals per phase
enum : int {
    TB_FULL = 0,                    // [kTcSlots] piece landed (1 + bytes)
    TB_EMPTY = TB_FULL + kTcSlots,  // [kTcSlots] MMAs reading the piece done (commit)
    TB_QROWS = TB_EMPTY + kTcSlots, // q rows of a run staged (8 softmax warps)
    TB_PROJ,                        // projection done (commit)
    TB_QT,                          // q~ staged (8)
    TB_SFULL,                       // [2] score tile done (commit)
    TB_PREADY = TB_SFULL + 2,       // [2] p tile written (8)
    TB_PVDONE = TB_PREADY + 2,      // [2] value products of that p tile done (commit)
    TB_VDONE = TB_PVDONE + 2,       // every value product of a segment done (commit)
    TB_VSTAGED,                     // v~ hi, lo written for the back-projection (8)
    TB_BPDONE,                      // back-projection done (commit)
    TB_FIN,                         // every MMA of the block done (commit)
    TB_NBAR
};

template <int D>
struct TcLay {
    static constexpr int kQ = kTcSlots * kTcSlot;                 // after the ring: q rows, cores [16 row groups][D/8]
    static constexpr int kQt = kQ + kTcRows * D * 2;              // q~ hi, then lo: cores [16][D/8] each
    static constexpr int kQtHalf = kTcRows * D * 2;
    static constexpr int kBar = kQt + 2 * kQtHalf;
    static constexpr int kX = kBar + TB_NBAR * 8;                 // pair exchange: maxima float [2][4 quarters][2][32],
    static constexpr int kFlag = kX + (2 * 4 * 2 + 4) * 32 * 4;   //   then row sums [4][32]; abort flag, tensor-memory base
    static constexpr int kTotal = kFlag + 16;
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
// D (+)= A B with A and B in shared memory
__device__ __forceinline__ void mma_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t id, bool acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(id), "r"((int)acc));
}
// D (+)= A B with A in tensor memory (row m on lane m, two bf16 a column)
__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a, uint64_t b, uint32_t id, bool acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
        "r"(a), "l"(b), "r"(id), "r"((int)acc));
}
// N products into one accumulator, unrolled: step k reads A at a + k a_step
// and B at b + k b_step (descriptor units of 16 bytes; tensor-memory A: 8
// columns = 16 bf16 a step); step 0 overwrites D unless acc0.
template <int N>
__device__ __forceinline__ void seq_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t a_step, uint32_t b_step,
                                       uint32_t id, bool acc0)
{
#pragma unroll
    for (int k = 0; k < N; ++k) mma_ss(d, a + (uint64_t)(k * a_step), b + (uint64_t)(k * b_step), id, k > 0 || acc0);
}
template <int N>
__device__ __forceinline__ void seq_ts(uint32_t d, uint32_t a, uint64_t b, uint32_t b_step, uint32_t id, bool acc0)
{
#pragma unroll
    for (int k = 0; k < N; ++k) mma_ts(d, a + 8u * k, b + (uint64_t)(k * b_step), id, k > 0 || acc0);
}
// f(integral_constant<int, n>) for a runtime n in 1..8
template <class F>
__device__ __forceinline__ void steps(int n, F &&f)
{
    switch (n) {
    case 1: f(std::integral_constant<int, 1>{}); break;
    case 2: f(std::integral_constant<int, 2>{}); break;
    case 3: f(std::integral_constant<int, 3>{}); break;
    case 4: f(std::integral_constant<int, 4>{}); break;
    case 5: f(std::integral_constant<int, 5>{}); break;
    case 6: f(std::integral_constant<int, 6>{}); break;
    case 7: f(std::integral_constant<int, 7>{}); break;
    default: f(std::integral_constant<int, 8>{}); break;
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
// 16 consecutive 32-bit columns of this warp's 32 lanes (no wait)
__device__ __forceinline__ void ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}
__device__ __forceinline__ void ld16f(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    ld16(taddr, r);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void st8(uint32_t taddr, const uint32_t *r)
{
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]),
                 "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                 : "memory");
}
__device__ __forceinline__ void st16(uint32_t taddr, const uint32_t *r)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}
__device__ __forceinline__ void wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// The 16-lane shapes: threads 0-15 access lanes base .. base + 15 at the
// address's column, threads 16-31 the same lanes OFF columns further.
template <int OFF>
__device__ __forceinline__ void ld16x2(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16], %17;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr), "n"(OFF)
        : "memory");
}
template <int OFF>
__device__ __forceinline__ void ld16x2f(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    ld16x2<OFF>(taddr, r);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
template <int OFF>
__device__ __forceinline__ void st8x2(uint32_t taddr, const uint32_t *r)
{
    asm volatile("tcgen05.st.sync.aligned.16x32bx2.x8.b32 [%0], %9, {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]),
                 "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "n"(OFF)
                 : "memory");
}
template <int OFF>
__device__ __forceinline__ void st16x2(uint32_t taddr, const uint32_t *r)
{
    asm volatile(
        "tcgen05.st.sync.aligned.16x32bx2.x16.b32 [%0], %17, {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "n"(OFF)
        : "memory");
}
}  // namespace tc

// Packed fp32 pairs (one 64-bit register pair; x in the low half): the
// paired add and subtract round each lane as the scalar instructions do.
__device__ __forceinline__ uint64_t f2(float x, float y)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
    return r;
}
__device__ __forceinline__ void f2get(uint64_t r, float &x, float &y) { asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(r)); }
__device__ __forceinline__ uint64_t f2add(uint64_t a, uint64_t b)
{
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f2sub(uint64_t a, uint64_t b)
{
    uint64_t r;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ float max3(float a, float b, float c)
{
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}
// The maximum of N values by a tree of three-input maxima.
template <int N>
__device__ __forceinline__ float max_tree(const float *v)
{
    if constexpr (N == 1) {
        return v[0];
    } else if constexpr (N == 2) {
        return fmaxf(v[0], v[1]);
    } else {
        constexpr int M = (N + 2) / 3;
        float t[M];
#pragma unroll
        for (int i = 0; i < N / 3; ++i) t[i] = max3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
        if constexpr (N % 3 == 2) t[M - 1] = fmaxf(v[N - 2], v[N - 1]);
        if constexpr (N % 3 == 1) t[M - 1] = v[N - 1];
        return max_tree<M>(t);
    }
}

// Two fp32 values as a bf16x2 "hi" (each truncated to its leading 8
// significant bits: the top half of its bits) and the bf16x2 of their
// residuals (truncated the same way): x = hi + lo to within 2^-15 of |x|,
// in five integer and paired-add operations.  Low half = x0.
__device__ __forceinline__ void split2(float x0, float x1, uint32_t &hi, uint32_t &lo)
{
    const uint32_t u0 = __float_as_uint(x0), u1 = __float_as_uint(x1);
    float r0, r1;
    f2get(f2sub(f2(x0, x1), f2(__uint_as_float(u0 & 0xffff0000u), __uint_as_float(u1 & 0xffff0000u))), r0, r1);
    hi = __byte_perm(u0, u1, 0x7632);
    lo = __byte_perm(__float_as_uint(r0), __float_as_uint(r1), 0x7632);
}

// 16 fp32 values of one row as bf16 hi + lo into two K-major cores each
// (columns 8c .. 8c + 15 of the row): hi cores at `hi`, hi + 128, lo cores at
// `lo`, lo + 128 (each address already at the row's 16-byte line).
__device__ __forceinline__ void put16(uint8_t *hi, uint8_t *lo, const float (&x)[16])
{
    uint32_t h[8], l[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) split2(x[2 * j], x[2 * j + 1], h[j], l[j]);
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

// What a segment (tokens [t0, t1) of one entry) needs, as the producer, the
// MMA issuer and the softmax walk it.
struct SegPlan {
    int64_t ck, pk, cv, pv;  // packed byte offsets (C at token 0 of the entry)
    int n8;                  // entry tokens rounded up to 8
    int rk, rv, rk8, rv8;    // ranks and rank 8-groups
    int nk16, nv16;          // 16-rank steps
    int g, t0, t1;
    int ntiles, tpp, nc;     // 64-token tiles, tiles per C piece, C pieces
    bool first_of_run, last_of_run;
    int slot;                // run record slot
};

__device__ __forceinline__ SegPlan seg_plan(const TcSegDev &sd)
{
    SegPlan q;
    q.ck = sd.ck;
    q.pk = sd.pk;
    q.cv = sd.cv;
    q.pv = sd.pv;
    q.n8 = (sd.n + 7) & ~7;
    q.rk = sd.rk;
    q.rv = sd.rv;
    q.rk8 = (sd.rk + 7) / 8;
    q.rv8 = (sd.rv + 7) / 8;
    q.nk16 = (q.rk8 + 1) / 2;
    q.nv16 = (q.rv8 + 1) / 2;
    q.g = sd.g;
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

// The segments of a share, each role reading them two ahead of use (a
// segment's record is one 64-byte load whose latency the walk hides).
struct SegWalk {
    const TcSegDev *segs;
    int end;
    TcSegDev cur, next, after;  // segments s, s + 1, s + 2 once at(s) was called
    __device__ void start(const TcSegDev *sg, int s0, int s1)
    {
        segs = sg;
        end = s1;
        if (s0 < s1) next = segs[s0];
        if (s0 + 1 < s1) after = segs[s0 + 1];
    }
    // move to segment s (called for s = s_begin, s_begin + 1, ... in order)
    __device__ void at(int s)
    {
        cur = next;
        next = after;
        if (s + 2 < end) after = segs[s + 2];
    }
};

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
    // zero the ring, q rows and q~: every later read past a piece's data
    // (rank and token padding of the products) sees finite values
    for (int i = tid; i < L::kBar / 16; i += kTcThreads) reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
    if (tid == 0) {
        for (int i = 0; i < kTcSlots; ++i) {
            mbar_init(bar(TB_FULL + i), 1);
            mbar_init(bar(TB_EMPTY + i), 1);
        }
        mbar_init(bar(TB_QROWS), 8);
        mbar_init(bar(TB_PROJ), 1);
        mbar_init(bar(TB_QT), 8);
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(TB_SFULL + i), 1);
            mbar_init(bar(TB_PREADY + i), 8);
            mbar_init(bar(TB_PVDONE + i), 1);
        }
        mbar_init(bar(TB_VDONE), 1);
        mbar_init(bar(TB_VSTAGED), 8);
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
            // order: P^K of the first segment; then per segment the next
            // segment's P^K (its projection goes ahead), the C pieces, P^V
            auto issue_pk = [&](const SegPlan &q) {
                if (q.rk > 0)
                    ok = issue([&](uint32_t dst, uint32_t b) {
                        const uint32_t bytes = (uint32_t)q.rk8 * D * 16;
                        mbar_arrive_tx(b, bytes);
                        bulk_g2s(dst, p.packed + q.pk, bytes, b);
                    });
            };
            SegWalk w;
            w.start(p.tc_segs, s_begin, s_end);
            for (int s = s_begin; ok && s < s_end; ++s) {
                w.at(s);
                const SegPlan q = seg_plan(w.cur);
                if (s == s_begin) issue_pk(q);
                if (ok && s + 1 < s_end) issue_pk(seg_plan(w.next));
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
        // The whole warp walks the schedule (every value warp-uniform) and
        // one elected lane issues the products and their commits: issuing
        // from a converged warp keeps the tensor pipe fed, where a lone
        // lane branching between products left it idle most of the time.
        pdl_wait();
        int n = 0;      // pieces consumed (in producer order)
        int krun = 0;   // runs whose q rows were waited for
        bool ok = true;
        auto wait = [&](int b, int parity) {
            ok = __all_sync(0xffffffffu, ok && tc_wait(bar(b), (uint32_t)parity & 1u, p.status, abort_flag));
            tc::fence_after();
        };
        // f() on one elected lane (always lane 0: the warp is converged)
        auto on_one = [&](auto &&f) {
            uint32_t pred;
            asm volatile("{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\tselp.u32 %0, 1, 0, e;\n\t}" : "=r"(pred));
            if (pred) f();
            __syncwarp();
        };
        auto take = [&](int &slot) {
            slot = n % kTcSlots;
            wait(TB_FULL + slot, n / kTcSlots);
            ++n;
            return sbase + (uint32_t)slot * kTcSlot;
        };
        const uint32_t q_u = sbase + L::kQ, qt_u = sbase + L::kQt;
        // projection of segment q (waits for the run's q rows first)
        auto project = [&](const SegPlan &q) {
            if (q.first_of_run) {
                wait(TB_QROWS, krun);
                ++krun;
            }
            int sl = 0;
            uint32_t pk = 0;
            if (q.rk > 0) pk = take(sl);
            const bool go = ok;
            on_one([&] {
                if (q.rk > 0) {
                    if (go)
                        tc::seq_ss<D / 16>(tmem + kColQ, tc::sdesc(q_u, 128, DG * 128), tc::sdesc(pk, 128, DG * 128),
                                           16, 16, tc::idesc(false, false, 16 * q.nk16), false);
                    tc::commit(bar(TB_EMPTY + sl));
                }
                tc::commit(bar(TB_PROJ));
            });
        };
        // the back-projection of a segment, issued once the next segment's
        // first score products are on their way
        SegPlan bq = {};
        int bp_slot = -1, bp_k = 0;
        uint32_t bp_u = 0;
        bool o_acc = false;  // O already holds part of the run of the pending back-projection
        auto back_project = [&]() {
            wait(TB_VSTAGED, bp_k);
            const bool go = ok && bq.rv > 0, acc = o_acc;
            on_one([&] {
                if (go) {
                    // O += v~ P^V: A = v~ hi, then lo (tensor memory), K = 16 nv16 ranks, N = d
                    const uint32_t id = tc::idesc(false, true, D);
                    const uint64_t bd = tc::sdesc(bp_u, DG * 128, 128);
                    tc::steps(bq.nv16, [&](auto nc) {
                        constexpr int N = decltype(nc)::value;
                        tc::seq_ts<N>(tmem + kColO, tmem + kColV, bd, (2 * DG * 128) >> 4, id, acc);
                        tc::seq_ts<N>(tmem + kColO, tmem + kColV + 64, bd, (2 * DG * 128) >> 4, id, true);
                    });
                }
                tc::commit(bar(TB_BPDONE));
                if (bq.rv > 0) tc::commit(bar(TB_EMPTY + bp_slot));
            });
            if (go) o_acc = true;
        };
        // C pieces of the current segment, taken in order by the score
        // products and released by the value products: at most two are live
        // (tiles j + 1 and j + 2 once tile j's values are issued)
        struct Piece {
            uint32_t base, cvb;
            int slot;
        };
        Piece pc[2] = {};
        int kseg = 0, J = 0;
        SegWalk w;
        w.start(p.tc_segs, s_begin, s_end);
        if (s_begin < s_end) project(seg_plan(p.tc_segs[s_begin]));
        for (int s = s_begin; ok && s < s_end; ++s, ++kseg) {
            w.at(s);
            const SegPlan q = seg_plan(w.cur);
            const int J0 = J;
            // this segment's q~ is staged: the next segment's projection (its
            // q rows and P^K come first)
            wait(TB_QT, kseg);
            if (ok && s + 1 < s_end) project(seg_plan(w.next));
            // per-segment constants of the products (descriptors without
            // their address field; a 64-token tile of C^K and of C^V)
            const uint32_t kstride = 8u * q.rk8 * 128, vstride = 8u * q.rv8 * 128;
            const uint64_t bdS = tc::sdesc(0, 128, q.rk8 * 128), bdV = tc::sdesc(0, q.rv8 * 128, 128);
            const uint64_t aS_hi = tc::sdesc(qt_u, 128, DG * 128), aS_lo = tc::sdesc(qt_u + L::kQtHalf, 128, DG * 128);
            const uint32_t idS = tc::idesc(false, false, kTcTok), idV = tc::idesc(false, true, 16 * q.nv16);
            const uint32_t vkstep = (2u * q.rv8 * 128) >> 4;
            // pieces by counters: the score side opens them (tile s_in of
            // piece s_piece), the value side releases them (v_in of v_piece)
            int s_piece = -1, s_in = q.tpp - 1, v_piece = 0, v_in = 0;
            // the whole tile loop for a compile-time count of 16-rank score
            // steps (no per-tile dispatch)
            tc::steps(q.nk16, [&](auto nkc) {
                constexpr int NK = decltype(nkc)::value;
                // the score product of tile j into buffer (J0 + j) & 1 (after
                // the value product that read that buffer's last p tile, by
                // issue order)
                auto score = [&](int j) {
                    if (q.nc > 0 && ++s_in == q.tpp) {
                        s_in = 0;
                        ++s_piece;
                        Piece &x = pc[s_piece & 1];
                        x.base = take(x.slot);
                        int a, rows;
                        c_piece_rows(q, s_piece, a, rows);
                        x.cvb = x.base + (uint32_t)rows * q.rk8 * 16;
                    }
                    const int b = (J0 + j) & 1;
                    const bool go = ok && q.rk > 0;
                    const uint64_t bd = bdS | (uint64_t)(((pc[s_piece & 1].base + (uint32_t)s_in * kstride) >> 4) & 0x3FFF);
                    on_one([&] {
                        if (go) {
                            tc::seq_ss<NK>(tmem + kColS + kTcTok * b, aS_hi, bd, 16, 16, idS, false);
                            tc::seq_ss<NK>(tmem + kColS + kTcTok * b, aS_lo, bd, 16, 16, idS, true);
                        }
                        tc::commit(bar(TB_SFULL + b));
                    });
                };
                // this segment's first two score products, then the previous
                // segment's back-projection (before this segment's first value
                // product overwrites v~)
                if (ok) score(0);
                if (ok && q.ntiles > 1) score(1);
                if (kseg > 0) back_project();
                if (q.first_of_run) o_acc = false;
                for (int j = 0; ok && j < q.ntiles; ++j) {
                    const int Jt = J0 + j, b = Jt & 1;
                    wait(TB_PREADY + b, Jt >> 1);
                    const Piece x = pc[v_piece & 1];
                    const bool go = ok && q.rv > 0;
                    const bool release = q.nc > 0 && (v_in == q.tpp - 1 || j == q.ntiles - 1);
                    const uint64_t bd = bdV | (uint64_t)(((x.cvb + (uint32_t)v_in * vstride) >> 4) & 0x3FFF);
                    on_one([&] {
                        if (go) {
                            // v~ += p C^V: A = p hi, then lo (tensor memory), K = 64 tokens
                            const uint32_t pa = tmem + kColS + kTcTok * b;
                            tc::seq_ts<kTcTok / 16>(tmem + kColV, pa, bd, vkstep, idV, j > 0);
                            tc::seq_ts<kTcTok / 16>(tmem + kColV, pa + kTcTok / 2, bd, vkstep, idV, true);
                        }
                        tc::commit(bar(TB_PVDONE + b));
                        // the last tile of a piece releases its slot
                        if (release) tc::commit(bar(TB_EMPTY + x.slot));
                    });
                    if (++v_in == q.tpp) {
                        v_in = 0;
                        ++v_piece;
                    }
                    if (ok && j + 2 < q.ntiles) score(j + 2);
                }
            });
            J = J0 + q.ntiles;
            on_one([&] { tc::commit(bar(TB_VDONE)); });
            // this segment's back-projection waits for the next one's
            // projection and first score products
            bq = q;
            bp_k = kseg;
            if (q.rv > 0) bp_u = take(bp_slot);
        }
        if (ok && kseg > 0) back_project();
        on_one([&] { tc::commit(bar(TB_FIN)); });
        // (not given up on an abort: the tensor memory is released after it)
        mbar_wait(bar(TB_FIN), 0, p.status);
        tc::fence_after();
    } else {
        // ------------------------------------------------ softmax
        // Warps 2..9, two per tensor-memory lane quarter: the pair (half 0
        // and 1) shares the quarter's rows and splits every tile's 64
        // columns, every rank chunk and the head dimension; a pair meets
        // through a named barrier once per tile (the row maximum).  A tile
        // of at most 64 rows is spread 16 rows per quarter (row r on lane
        // 32 (r / 16) + r % 16, the other lanes hold zero rows), so that
        // all four sub-partitions share its softmax: a warp then reaches its
        // 16 lanes with the 16-lane shapes, threads 16-31 taking the second
        // half of the warp's columns.  Only a call of one such tile spreads:
        // beside full tiles of the same shares (which read the same pieces)
        // a spread tile gained nothing and the full ones slowed down (76 to
        // 81 us a block on the batch-64 layer, against 421 to 377 us for the
        // one tile of the 56-row, 1M-token layer).
        pdl_wait();  // q and the accumulators belong to the preceding grids until here
        const bool spread = p.tc_ntile == 1 && p.rows_g <= kTcRows / 2;
        auto role = [&](auto spc) {
            constexpr bool SP = decltype(spc)::value;
            const int quad = warp & 3, half = (warp - 2) >> 2;
            const int u = SP ? lane >> 4 : 0;           // SP: which 16 of the warp's 32 columns
            const int ts = SP ? lane & 15 : lane;       // the thread's row within the quarter
            const int rl = (SP ? 16 : 32) * quad + ts;  // row within the tile
            const int pos = 32 * quad + ts;             // its tensor-memory lane (and A-operand row)
            const int row = tile * kTcRows + rl;        // the KV head's query row (batch x heads)
            const bool row_ok = row < p.rows_g;
            const uint32_t tl = tmem + ((uint32_t)(32 * quad) << 16);
            uint8_t *q_s = smem + L::kQ, *qt_s = smem + L::kQt;
            float *xch = reinterpret_cast<float *>(smem + L::kX);  // maxima [2][4][2][32], row sums [4][32]
            const int rg8 = pos >> 3, r8 = pos & 7;     // core row group and row within the core (r8 = row % 8)
            constexpr int kHalfTok = kTcTok / 2;        // columns of a tile per warp
            constexpr int kCols = SP ? kHalfTok / 2 : kHalfTok;  // ... per thread
            int J = 0, kseg = 0, kproj = 0, bp_waited = 0;
            bool ok = true;
            float m = -INFINITY, l = 0.f;             // l: this warp's columns only
            bool o_written = false, first_tile = true;
            uint32_t ref = 0u;
            auto arrive = [&](int b) {
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(b));
            };
            auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + quad) : "memory"); };
            // the warp-collective tensor-memory accesses after a wait need every
            // lane to agree on its outcome
            auto wwait = [&](int b, int parity) {
                ok = __all_sync(0xffffffffu, ok && tc_wait(bar(b), (uint32_t)parity & 1u, p.status, abort_flag));
                tc::fence_after();
            };
            // back-projections done up to segment k (in phase order)
            auto wait_bp_upto = [&](int k) {
                while (bp_waited <= k) {
                    wwait(TB_BPDONE, bp_waited);
                    ++bp_waited;
                }
            };
            // a run's q rows as the projection's A operand (this thread's share
            // of the columns)
            auto write_qrows = [&](const SegPlan &q) {
                const uint4 *qr = reinterpret_cast<const uint4 *>(
                    p.q + ((int64_t)(row / p.G) * p.hq + q.g * p.G + row % p.G) * D);
                constexpr int kParts = SP ? 4 : 2;
                const int part = SP ? 2 * half + u : half;
    #pragma unroll 4
                for (int c = part * (DG / kParts); c < (part + 1) * (DG / kParts); ++c) {
                    const uint4 v = row_ok ? __ldcg(qr + c) : make_uint4(0u, 0u, 0u, 0u);
                    *reinterpret_cast<uint4 *>(q_s + (rg8 * DG + c) * 128 + r8 * 16) = v;
                }
                tc::fence_proxy();
                arrive(TB_QROWS);
            };
            // segment s's q~ = scale log2(e) Q P^K^T as hi and lo A operands in
            // shared memory (rank chunks of this warp's parity; ranks past the
            // rank: zero), then the next run's q rows if segment s + 1 starts one
            // (its projection is issued as soon as q~ is staged)
            auto prepare = [&](int s, const TcSegDev &sd, const TcSegDev &sd_next) {
                const SegPlan q = seg_plan(sd);
                wwait(TB_PROJ, kproj++);
                if (ok) {
                    // rank chunks of 16: SP, chunk pair cp (of this warp's
                    // parity) gives the thread chunk 2 cp + u
    #pragma unroll 1
                    for (int cc = half; (SP ? 2 * cc : cc) < q.nk16; cc += 2) {
                        float v[16];
                        int c = cc;
                        if constexpr (SP) {
                            tc::ld16x2f<16>(tl + kColQ + 32 * cc, v);
                            c = 2 * cc + u;
                        } else {
                            tc::ld16f(tl + kColQ + 16 * cc, v);
                        }
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
                if (s + 1 < s_end) {
                    const SegPlan qn = seg_plan(sd_next);
                    if (qn.first_of_run) write_qrows(qn);
                }
            };
            SegWalk w;
            w.start(p.tc_segs, s_begin, s_end);
            if (s_begin < s_end) {
                const TcSegDev first = p.tc_segs[s_begin];
                write_qrows(seg_plan(first));
                prepare(s_begin, first, s_begin + 1 < s_end ? p.tc_segs[s_begin + 1] : first);
            }
            for (int s = s_begin; s < s_end; ++s, ++kseg) {
                w.at(s);
                const SegPlan q = seg_plan(w.cur);
                const int g = q.g;
                if (q.first_of_run) {
                    m = -INFINITY;
                    l = 0.f;
                    o_written = false;
                    first_tile = true;
                }
                const int ntok = q.t1 - q.t0;
    #pragma unroll 1
                for (int j = 0; j < q.ntiles; ++j, ++J) {
                    const int b = J & 1;
                    const uint32_t sb = tl + kColS + kTcTok * b;
                    wwait(TB_SFULL + b, J >> 1);
                    float sv[kCols];
                    if (ok && q.rk > 0) {
                        if constexpr (SP) {
                            tc::ld16x2f<16>(sb + kHalfTok * half, sv);
                            tc::wait_ld();
                        } else {
                            float v0[16], v1[16];
                            tc::ld16f(sb + kHalfTok * half, v0);
                            tc::ld16f(sb + kHalfTok * half + 16, v1);
                            tc::wait_ld();
    #pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                sv[i] = v0[i];
                                sv[16 + i] = v1[i];
                            }
                        }
                    } else {
    #pragma unroll
                        for (int i = 0; i < kCols; ++i) sv[i] = 0.f;
                    }
                    // this thread's valid columns
                    const int nvalid = min(kTcTok, ntok - kTcTok * j) - kHalfTok * half - kCols * u;
                    if (nvalid < kCols) {
    #pragma unroll
                        for (int i = 0; i < kCols; ++i) sv[i] = i < nvalid ? sv[i] : -INFINITY;
                    }
                    // the row maximum of the tile: a tree over this warp's columns,
                    // then the pair's two halves through shared memory (both
                    // warps have read their scores before either overwrites the
                    // tile with p)
                    float tmax = max_tree<kCols>(sv);
                    if constexpr (SP) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 16));
                    float *xb = xch + ((J & 1) * 4 + quad) * 64;
                    xb[half * 32 + ts] = tmax;
                    pair_sync();
                    const float mx = fmaxf(tmax, xb[(1 - half) * 32 + ts]);
                    // lazy rescale: the reference moves only when a score passes it
                    // by kLazyTc; V~ and O, already summed against the old one,
                    // are multiplied by 2^(m_old - m_new) in tensor memory (the
                    // pair splits the rank and head-dimension chunks)
                    const bool need = mx > m + kLazyTc;
                    if (__any_sync(0xffffffffu, need)) {
                        const float mn = need ? mx : m;
                        const float alpha = need ? exp2_diff(m, mn) : 1.f;
                        if (j > 0) {
                            // the value products of tile j - 1 (and every earlier
                            // product) must be done
                            const int Jp = J - 1;
                            wwait(TB_PVDONE + (Jp & 1), Jp >> 1);
                            if (ok && q.rv > 0) {
    #pragma unroll 1
                                for (int c = half; (SP ? 2 * c : c) < q.nv16; c += 2) {
                                    uint32_t r[16];
                                    if constexpr (SP) tc::ld16x2<16>(tl + kColV + 32 * c, r); else tc::ld16(tl + kColV + 16 * c, r);
                                    tc::wait_ld();
    #pragma unroll
                                    for (int i = 0; i < 16; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
                                    if constexpr (SP) tc::st16x2<16>(tl + kColV + 32 * c, r); else tc::st16(tl + kColV + 16 * c, r);
                                }
                            }
                        }
                        if (o_written) {
                            wait_bp_upto(kseg - 1);  // every back-projection of the run is done
                            if (ok) {
    #pragma unroll 1
                                for (int c = half; c < (SP ? D / 32 : D / 16); c += 2) {
                                    uint32_t r[16];
                                    if constexpr (SP) tc::ld16x2<16>(tl + kColO + 32 * c, r); else tc::ld16(tl + kColO + 16 * c, r);
                                    tc::wait_ld();
    #pragma unroll
                                    for (int i = 0; i < 16; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
                                    if constexpr (SP) tc::st16x2<16>(tl + kColO + 32 * c, r); else tc::st16(tl + kColO + 16 * c, r);
                                }
                            }
                        }
                        tc::wait_st();
                        l *= alpha;
                        m = mn;
                    }
                    if (first_tile) {
                        ref = publish_ref(p, g, row, row_ok, u, m);  // (SP: the thread with u = 0)
                        if constexpr (SP) ref = __shfl_sync(0xffffffffu, ref, ts);
                        first_tile = false;
                    }
                    // p = 2^(s - m) of this warp's columns as bf16 hi | lo over the
                    // score tile (hi in columns [0, 32), lo in [32, 64))
                    uint32_t ph[kCols / 2], pl[kCols / 2];
                    uint64_t t2[kCols / 2];  // pairs of p, then their pairwise sums
                    const uint64_t m2 = f2(m, m);
    #pragma unroll
                    for (int i = 0; i < kCols / 2; ++i) {
                        float d0, d1;
                        f2get(f2sub(f2(sv[2 * i], sv[2 * i + 1]), m2), d0, d1);
                        const float p0 = ex2_approx(d0), p1 = ex2_approx(d1);  // masked: 0
                        t2[i] = f2(p0, p1);
                        split2(p0, p1, ph[i], pl[i]);
                    }
    #pragma unroll
                    for (int w = kCols / 4; w >= 1; w /= 2)
    #pragma unroll
                        for (int i = 0; i < w; ++i) t2[i] = f2add(t2[i], t2[i + w]);
                    {
                        float a, c;
                        f2get(t2[0], a, c);
                        l += a + c;
                    }
                    if constexpr (SP) {
                        tc::st8x2<8>(sb + (kHalfTok / 2) * half, ph);
                        tc::st8x2<8>(sb + kTcTok / 2 + (kHalfTok / 2) * half, pl);
                    } else {
                        tc::st16(sb + (kHalfTok / 2) * half, ph);
                        tc::st16(sb + kTcTok / 2 + (kHalfTok / 2) * half, pl);
                    }
                    tc::wait_st();
                    tc::fence_before();
                    arrive(TB_PREADY + b);
                }
                // the next segment's q~ (its projection went ahead), then this
                // segment's v~ as the back-projection's hi and lo A operands, in
                // place in tensor memory (hi at +0, lo at +64; ranks past the
                // rank: zero): both warps of the pair read their chunks before
                // either writes
                if (s + 1 < s_end) prepare(s + 1, w.next, w.after);
                wwait(TB_VDONE, kseg);
                if (q.rv > 0) {
                    // (the pair barrier runs in both warps whatever ok says)
                    // rank chunks of 16 (SP: chunk pairs, the thread's chunk 2 cc + u)
                    constexpr int kNC = SP ? D / 64 : D / 32;  // chunks (SP: pairs) per warp
                    uint32_t vh[8 * kNC], vl[8 * kNC];
    #pragma unroll
                    for (int k = 0; k < kNC; ++k) {
                        const int cc = 2 * k + half, c = SP ? 2 * cc + u : cc;
                        if (ok && (SP ? 2 * cc : cc) < q.nv16) {
                            float v[16];
                            if constexpr (SP) tc::ld16x2f<16>(tl + kColV + 32 * cc, v); else tc::ld16f(tl + kColV + 16 * cc, v);
                            tc::wait_ld();
    #pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const float x0 = 16 * c + 2 * i < q.rv ? v[2 * i] : 0.f;
                                const float x1 = 16 * c + 2 * i + 1 < q.rv ? v[2 * i + 1] : 0.f;
                                split2(x0, x1, vh[8 * k + i], vl[8 * k + i]);
                            }
                        }
                    }
                    pair_sync();
    #pragma unroll
                    for (int k = 0; k < kNC; ++k) {
                        const int cc = 2 * k + half;
                        if (ok && (SP ? 2 * cc : cc) < q.nv16) {
                            if constexpr (SP) {
                                tc::st8x2<8>(tl + kColV + 16 * cc, vh + 8 * k);
                                tc::st8x2<8>(tl + kColV + 64 + 16 * cc, vl + 8 * k);
                            } else {
                                tc::st8(tl + kColV + 8 * cc, vh + 8 * k);
                                tc::st8(tl + kColV + 64 + 8 * cc, vl + 8 * k);
                            }
                        }
                    }
                    tc::wait_st();
                }
                tc::fence_before();
                // the previous segment's back-projection is done before this
                // one's can be (the phase order of its barrier)
                wait_bp_upto(kseg - 1);
                arrive(TB_VSTAGED);
                if (q.rv > 0) o_written = true;
                if (q.last_of_run) {
                    wait_bp_upto(kseg);
                    // ---- the run's result into the accumulators of KV head g
                    // (or, for a row group with an outlier maximum, as a record);
                    // the pair adds its row sums, each warp its half of O
                    float *xl = xch + 2 * 4 * 2 * 32 + quad * 32;
                    float lw = l;
                    if constexpr (SP) lw += __shfl_xor_sync(0xffffffffu, lw, 16);
                    if (half == 1) xl[ts] = lw;
                    pair_sync();
                    const float lsum = half == 0 ? lw + xl[ts] : 0.f;  // used by half 0
                    const float Mref = ref ? ref_dec(ref) : m;
                    const bool outlier = row_ok && m - Mref > kDirectMax;
                    const uint32_t votes = __ballot_sync(0xffffffffu, outlier);
                    const bool direct = ((votes >> (ts & ~7)) & 0xffu) == 0u;  // the row's group of 8
                    const int rgg = row >> 3;
                    const int64_t rec_idx = (int64_t)q.slot * p.nrg + rgg;
                    float *rec = p.rec + rec_idx * (8 * D + kRecFloatsExtra);
                    const float f = row_ok && direct ? ex2_approx(m - Mref) : 0.f;
                    float *arow = p.acc_o + ((int64_t)g * p.rows_max + row) * D;
                    if (ok) {
    #pragma unroll 1
                        for (int cc = half; cc < (SP ? D / 32 : D / 16); cc += 2) {
                            float o[16];
                            const int c = SP ? 2 * cc + u : cc;  // this thread's 16 columns
                            if (o_written) {
                                if constexpr (SP) tc::ld16x2f<16>(tl + kColO + 32 * cc, o); else tc::ld16f(tl + kColO + 16 * cc, o);
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
                        if (row_ok && half == 0 && u == 0) {
                            if (direct) {
                                atomicAdd(p.acc_l + (int64_t)g * p.rows_max + row, f * lsum);
                            } else {
                                __stcg(rec + 8 * D + r8, m);
                                __stcg(rec + 8 * D + 8 + r8, lsum);
                            }
                        }
                        // one lane per row group lists an outlier record
                        if (!direct && half == 0 && u == 0 && r8 == 0 && row_ok) {
                            const int gr = g * p.nrg + rgg;
                            const uint32_t k = atomicAdd(p.ovf_cnt + gr, 1u);
                            __stcg(reinterpret_cast<int4 *>(p.ovf_list) + (int64_t)gr * p.list_cap + k,
                                   make_int4((int)rec_idx, 8 * rgg, min(8, p.rows_g - 8 * rgg), 0));
                        }
                    }
                    tc::fence_before();
                }
            }
        };
        if (spread) role(std::true_type{}); else role(std::false_type{});
    }
    // every MMA is done (the issuer waited for them) and every tensor-memory
    // access has completed: release the tensor memory
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
