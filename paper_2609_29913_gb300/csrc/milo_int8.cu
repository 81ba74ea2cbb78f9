// milo_int8.cu -- group-wise asymmetric INT8 storage of a packed arena (the
// "MILO + INT8" setting of Sec. 5.3, Table 2: asymmetric INT8 quantisation on
// top of the low-rank factors).
//
// A group is one 8x8 bf16 core of the packed arena (128 contiguous bytes: 8
// tokens x 8 ranks of a C factor, or 8 ranks x 8 columns of a P factor).  Per
// group: the minimum m (+0 for a zero), a step s = (max - m) / 255 in fp32
// rounded up to bf16 (so every code stays within 255), codes
// c = rint((x - m) * (1/s)) clamped to [0, 255] (0 when s = 0 or 1/s
// overflows), and the value read back
// bf16(m + s c) (s c is exact in fp32; one rounding for the sum, one to bf16).
// Codes keep the element order of the core (64 bytes per group); the
// parameters are one 32-bit word per group, m in the low half and s in the
// high half, both bf16 bit patterns.
//
// Both kernels stream: eight lanes per group (one 16-byte row of the core per
// lane), four groups per warp and step, a warp-uniform loop so the team
// shuffles always see the whole warp.  The dequantising kernel also reads
// codes from mapped pinned host memory (the offloaded INT8 prefix), where
// each lane keeps two groups' loads in flight to cover the link's latency.
#include <algorithm>

#include <cuda_bf16.h>

#include "milo_int8.cuh"
#include "milo_internal.h"

namespace milo {
namespace {

constexpr int kInt8Threads = 256;

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__global__ void __launch_bounds__(kInt8Threads) quant_kernel(const uint4 *__restrict__ src,
                                                             uint2 *__restrict__ codes,
                                                             uint32_t *__restrict__ params, int64_t groups)
{
    const int lane = threadIdx.x & 31, row = lane & 7, team = lane >> 3;
    const int64_t warp = ((int64_t)blockIdx.x * kInt8Threads + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * kInt8Threads) >> 5;
    for (int64_t g0 = 4 * warp; g0 < groups; g0 += 4 * nwarps) {
        const int64_t g = g0 + team;
        const bool live = g < groups;
        uint4 w = make_uint4(0, 0, 0, 0);
        if (live) w = src[g * 8 + row];
        float x[8] = {bf_lo(w.x), bf_hi(w.x), bf_lo(w.y), bf_hi(w.y),
                      bf_lo(w.z), bf_hi(w.z), bf_lo(w.w), bf_hi(w.w)};
        float lo = x[0], hi = x[0];
#pragma unroll
        for (int i = 1; i < 8; ++i) {
            lo = fminf(lo, x[i]);
            hi = fmaxf(hi, x[i]);
        }
#pragma unroll
        for (int off = 1; off < 8; off <<= 1) {
            lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, off));
            hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, off));
        }
        lo = __fadd_rn(lo, 0.f);  // -0 -> +0, so the stored m does not depend on which zero won
        hi = __fadd_rn(hi, 0.f);
        const uint32_t q = __float_as_uint(__fdiv_rn(__fsub_rn(hi, lo), 255.f));
        const uint32_t sb = (q >> 16) + ((q & 0xFFFFu) != 0u);   // round up to bf16
        const float s = __uint_as_float(sb << 16);
        float inv = __frcp_rn(s);
        if (!(s > 0.f) || isinf(inv)) inv = 0.f;  // s = 0 (or below 2^-128): every code 0
        uint32_t packed[2] = {0u, 0u};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            int c = __float2int_rn(__fmul_rn(__fsub_rn(x[i], lo), inv));
            c = min(max(c, 0), 255);
            packed[i >> 2] |= (uint32_t)c << (8 * (i & 3));
        }
        if (live) {
            codes[g * 8 + row] = make_uint2(packed[0], packed[1]);
            if (row == 0) params[g] = (__float_as_uint(lo) >> 16) | (sb << 16);
        }
    }
}

__global__ void __launch_bounds__(kInt8Threads) dequant_kernel(const uint2 *__restrict__ codes,
                                                               const uint32_t *__restrict__ params,
                                                               uint4 *__restrict__ dst, int64_t groups)
{
    const int lane = threadIdx.x & 31, row = lane & 7, team = lane >> 3;
    const int64_t warp = ((int64_t)blockIdx.x * kInt8Threads + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * kInt8Threads) >> 5;
    const int64_t step = 4 * nwarps;
    int64_t g = 4 * warp + team;
    // two groups per lane and step: both loads issued before either is used
    for (; g + step < groups; g += 2 * step) {
        const uint2 c0 = codes[g * 8 + row], c1 = codes[(g + step) * 8 + row];
        const uint32_t p0 = params[g], p1 = params[g + step];
        dst[g * 8 + row] = dequant_row(c0, p0);
        dst[(g + step) * 8 + row] = dequant_row(c1, p1);
    }
    if (g < groups) dst[g * 8 + row] = dequant_row(codes[g * 8 + row], params[g]);
}

// The read-back of a plan's arena: blocks over (entry, factor, slice of
// kPlanGroups cores) (grid E x 4 x slices: C^K, P^K, C^V, P^V), so each core
// knows which of its rows and columns are padding (ranks past r, tokens past
// n) and writes 0 there instead of m + s c: the staged arena then holds
// exactly the zero-padded read-back factors the decode kernels expect.  Each
// lane issues the loads of its four cores before converting any of them.
// (128-thread blocks: small enough in registers to run beside the decode
// grid's blocks of the layer before, which the staging overlaps)
constexpr int kPlanThreads = 128;
constexpr int kPlanUnroll = 4;
constexpr int kPlanGroups = (kPlanThreads / 8) * kPlanUnroll;   // cores per block

__global__ void __launch_bounds__(kPlanThreads) dequant_plan_kernel(const EntryDev *__restrict__ entries, int head_dim,
                                                                    const uint2 *__restrict__ codes,
                                                                    const uint32_t *__restrict__ params,
                                                                    uint4 *__restrict__ dst)
{
    const int f = blockIdx.y;
    const EntryDev ent = entries[blockIdx.x];
    const int r = (f < 2) ? ent.rk : ent.rv;
    const int r8 = (r + 7) & ~7;
    // C: rows = tokens (n), columns = ranks (r); P: rows = ranks (r), columns = head_dim
    const int cgs = ((f & 1) ? head_dim : r8) / 8;
    const int rgs = ((f & 1) ? r8 : ((ent.n + 7) & ~7)) / 8;
    const int total = rgs * cgs;
    const int base = blockIdx.z * kPlanGroups;
    if (base >= total) return;
    const int rows = (f & 1) ? r : ent.n;
    const int cols = (f & 1) ? head_dim : r;
    const int64_t off = (f == 0) ? ent.off_ck : (f == 1) ? ent.off_pk : (f == 2) ? ent.off_cv : ent.off_pv;
    const int64_t g0 = off / 128;
    const bool ragged = ((rows | cols) & 7) != 0;   // padding only when n or r is not a multiple of 8
    const int row = threadIdx.x & 7, team = threadIdx.x >> 3;
    uint2 c[kPlanUnroll];
    uint32_t pw[kPlanUnroll];
#pragma unroll
    for (int u = 0; u < kPlanUnroll; ++u) {
        const int t = base + team + u * (kPlanThreads / 8);
        if (t < total) {
            c[u] = codes[(g0 + t) * 8 + row];
            pw[u] = params[g0 + t];
        }
    }
#pragma unroll
    for (int u = 0; u < kPlanUnroll; ++u) {
        const int t = base + team + u * (kPlanThreads / 8);
        if (t >= total) break;
        uint4 v = dequant_row(c[u], pw[u]);
        int valid = 8;
        if (ragged) {
            const int tr = t / cgs, tc = t - tr * cgs;
            valid = (8 * tr + row < rows) ? min(8, cols - 8 * tc) : 0;
        }
        if (valid < 8) {
            uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (i >= valid) w[i >> 1] &= (i & 1) ? 0x0000FFFFu : 0xFFFF0000u;
            v = make_uint4(w[0], w[1], w[2], w[3]);
        }
        dst[(g0 + t) * 8 + row] = v;
    }
}

int int8_grid(int64_t groups, int blocks_per_sm)
{
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
    const int64_t want = (groups + (kInt8Threads / 8) - 1) / (kInt8Threads / 8);
    return (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sms * blocks_per_sm));
}

}  // namespace

cudaError_t launch_quant_int8(const void *packed, int64_t groups, void *codes, void *params, cudaStream_t stream)
{
    if (groups <= 0) return cudaSuccess;
    quant_kernel<<<int8_grid(groups, 8), kInt8Threads, 0, stream>>>(
        static_cast<const uint4 *>(packed), static_cast<uint2 *>(codes), static_cast<uint32_t *>(params), groups);
    return cudaGetLastError();
}

cudaError_t launch_dequant_int8(const void *codes, const void *params, int64_t groups, void *packed,
                                cudaStream_t stream)
{
    if (groups <= 0) return cudaSuccess;
    dequant_kernel<<<int8_grid(groups, 4), kInt8Threads, 0, stream>>>(
        static_cast<const uint2 *>(codes), static_cast<const uint32_t *>(params), static_cast<uint4 *>(packed), groups);
    return cudaGetLastError();
}

cudaError_t launch_dequant_plan_int8(const EntryDev *entries, int num_entries, int head_dim, int64_t max_factor_groups,
                                     const void *codes, const void *params, void *packed, cudaStream_t stream)
{
    if (num_entries <= 0 || max_factor_groups <= 0) return cudaSuccess;
    const int slices = (int)((max_factor_groups + kPlanGroups - 1) / kPlanGroups);
    dequant_plan_kernel<<<dim3(num_entries, 4, slices), kPlanThreads, 0, stream>>>(
        entries, head_dim, static_cast<const uint2 *>(codes), static_cast<const uint32_t *>(params),
        static_cast<uint4 *>(packed));
    return cudaGetLastError();
}

}  // namespace milo
