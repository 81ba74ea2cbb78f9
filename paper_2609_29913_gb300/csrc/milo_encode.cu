// milo_encode.cu -- the compression stage on the GPU (Alg. 1 Stage 1): for
// every block b and KV head g of a prefix, the SVD of its keys and of its
// values (Eq. 3), the rank allocation over the blocks of each (KV head, K or
// V) group (Eq. 6 by the greedy of Eq. 7), and the rank-r factors
// C = A Sigma (n x r) and P = B^T (r x d) written as bf16 into an arena laid
// out for milo_prefix_create.
//
//   spectrum_kernel  one block per (entry, K or V): the Gram matrix
//                    G = X^T X of the block's rows (bf16 inputs, fp32 sums),
//                    its eigenvalues and eigenvectors by cyclic Jacobi
//                    rotations in shared memory (the tournament order lets
//                    d/2 disjoint rotations run at once), sorted so that
//                    sigma_j = sqrt(lambda_j) is non-increasing.  G = B
//                    Sigma^2 B^T, so the eigenvectors are the right singular
//                    vectors.
//   allocate_kernel  one block per (KV head, K or V) group: every block
//                    first gets min(r_min, avail) units; the greedy then
//                    gives the remaining R_tot - sum units one at a time to
//                    the block whose next singular value has the largest
//                    gain log(1 + sigma^2 / eps^2), ties to the lowest block.
//                    The gain grows with sigma, and a block's next value is
//                    never above its previous one, so the greedy takes the
//                    U largest candidates sigma_{b,j} (j from avail-capped
//                    r_min to the cap) in the order (sigma descending, block,
//                    j); the kernel finds the U-th largest value tau by a
//                    binary search over the float bits (counting candidates
//                    above it) and breaks the ties at tau in (block, j)
//                    order.
//   factor_kernel    one block per (entry, K or V): C = X B_r (the rank-r
//                    columns of A Sigma) and P = B_r^T, both rounded to bf16.
//
// Everything is fp32 on CUDA cores: the stage runs once per prefix, and fp32
// keeps the allocation decisions to the precision the tests reproduce (the
// oracle's greedy, fed the same singular values, gives the same ranks).
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <vector>

#include "milo.h"
#include "milo_internal.h"

namespace milo {
namespace {

constexpr int kEncThreads = 256;
constexpr int kEncTok = 64;            // tokens per staged tile
constexpr int kJacobiMaxSweeps = 20;
constexpr float kJacobiTol = 1e-6f;    // off-diagonal Frobenius norm / total, to stop

struct EncParams {
    const uint16_t *k, *v;    // bf16 [N, Hkv, d]
    const int64_t *tok0;      // [nb] first token of each block
    const int32_t *blen;      // [nb]
    const int64_t *offs;      // [E][4] element offsets of C^K, P^K, C^V, P^V
    uint16_t *arena;          // bf16
    int32_t *rank_k, *rank_v; // [E]
    float *sigma;             // [2E][d]: entry e's keys at 2e, values at 2e + 1
    float *vt;                // [2E][d][d]: eigenvectors as rows, by sigma
    int32_t *status;          // device status word (0 ok)
    int nb, hkv, d;
    int r_min, r_max;
    int64_t budget_k, budget_v;
};

// Rows of the Gram matrix and of the rotation matrix in shared memory are
// D + 1 floats apart, so that a column of either (fixed column, rows apart)
// falls on distinct banks.
template <int D>
struct EncLay {
    static constexpr int kLd = D + 1;
    static constexpr int kG = 0;                          // [D][kLd] G, then the rotated G
    static constexpr int kV = kG + D * kLd * 4;           // [D][kLd] accumulated rotations
    static constexpr int kX = kV + D * kLd * 4;           // [kEncTok][D] fp32 tile of rows
    static constexpr int kRot = kX + kEncTok * D * 4;     // [D/2] (c, s) and [D/2] (p, q)
    static constexpr int kRed = kRot + (D / 2) * 16;      // reduction scratch
    static constexpr int kTotal = kRed + 64 * 4;
};

__device__ __forceinline__ float bf16f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ long long llmin(long long a, long long b) { return a < b ? a : b; }
__device__ __forceinline__ long long llmax(long long a, long long b) { return a > b ? a : b; }

// Tournament pairing for round r of n - 1 (n even): pair 0 is (n - 1, r),
// pair k > 0 is ((r + k) % (n - 1), (r - k + n - 1) % (n - 1)).
__device__ __forceinline__ void pair_of(int n, int r, int k, int &p, int &q)
{
    if (k == 0) {
        p = n - 1;
        q = r;
    } else {
        p = (r + k) % (n - 1);
        q = (r - k + n - 1) % (n - 1);
    }
    if (p > q) {
        const int t = p;
        p = q;
        q = t;
    }
}

template <int D>
__global__ void __launch_bounds__(kEncThreads, 1) spectrum_kernel(const EncParams p)
{
    using L = EncLay<D>;
    extern __shared__ __align__(16) uint8_t smem[];
    float *G = reinterpret_cast<float *>(smem + L::kG);
    float *V = reinterpret_cast<float *>(smem + L::kV);
    float *X = reinterpret_cast<float *>(smem + L::kX);
    float4 *rot = reinterpret_cast<float4 *>(smem + L::kRot);  // (c, s, p, q)
    float *red = reinterpret_cast<float *>(smem + L::kRed);
    const int tid = threadIdx.x;
    const int m = blockIdx.x;  // 2 e + side
    const int e = m >> 1, side = m & 1;
    const int b = e / p.hkv, g = e % p.hkv;
    const int n = p.blen[b];
    const uint16_t *src = (side ? p.v : p.k) + (p.tok0[b] * p.hkv + g) * (int64_t)D;
    const int64_t rstride = (int64_t)p.hkv * D;

    // ---- G = X^T X: thread (ti, tj) sums the T x T tile of rows T ti ..,
    // columns T tj .. (T = D / 16: 256 tiles)
    constexpr int T = D / 16;
    const int ti = tid / 16, tj = tid % 16;
    float acc[T][T];
#pragma unroll
    for (int a = 0; a < T; ++a)
#pragma unroll
        for (int c = 0; c < T; ++c) acc[a][c] = 0.f;
    for (int t0 = 0; t0 < n; t0 += kEncTok) {
        const int nt = min(kEncTok, n - t0);
        __syncthreads();
        for (int x = tid; x < kEncTok * D / 2; x += kEncThreads) {
            const int t = x / (D / 2), c = 2 * (x % (D / 2));
            float a = 0.f, bb = 0.f;
            if (t < nt) {
                const uint32_t w = *reinterpret_cast<const uint32_t *>(src + (int64_t)(t0 + t) * rstride + c);
                a = bf16f((uint16_t)(w & 0xffffu));
                bb = bf16f((uint16_t)(w >> 16));
            }
            X[t * D + c] = a;
            X[t * D + c + 1] = bb;
        }
        __syncthreads();
        for (int t = 0; t < nt; ++t) {
            float xa[T], xb[T];
#pragma unroll
            for (int a = 0; a < T; ++a) {
                xa[a] = X[t * D + T * ti + a];
                xb[a] = X[t * D + T * tj + a];
            }
#pragma unroll
            for (int a = 0; a < T; ++a)
#pragma unroll
                for (int c = 0; c < T; ++c) acc[a][c] = fmaf(xa[a], xb[c], acc[a][c]);
        }
    }
    // G, and a copy of it in this matrix's eigenvector slot (the eigenvalues
    // are read off at the end as Rayleigh quotients against it)
    float *g0 = p.vt + (int64_t)m * D * D;
#pragma unroll
    for (int a = 0; a < T; ++a)
#pragma unroll
        for (int c = 0; c < T; ++c) {
            G[(T * ti + a) * L::kLd + T * tj + c] = acc[a][c];
            g0[(T * ti + a) * D + T * tj + c] = acc[a][c];
        }
    for (int x = tid; x < D * D; x += kEncThreads) V[(x / D) * L::kLd + x % D] = (x / D == x % D) ? 1.f : 0.f;
    __syncthreads();

    // ---- cyclic Jacobi sweeps, D/2 disjoint rotations per round
    float total = 0.f;  // Frobenius norm^2 of G (kept by the rotations)
    for (int x = tid; x < D * D; x += kEncThreads) {
        const float y = G[(x / D) * L::kLd + x % D];
        total += y * y;
    }
    for (int o = 16; o; o >>= 1) total += __shfl_xor_sync(0xffffffffu, total, o);
    if ((tid & 31) == 0) red[tid >> 5] = total;
    __syncthreads();
    total = 0.f;
    for (int w = 0; w < kEncThreads / 32; ++w) total += red[w];
    __syncthreads();
    for (int sweep = 0; sweep < kJacobiMaxSweeps; ++sweep) {
        // off-diagonal norm^2
        float off = 0.f;
        for (int x = tid; x < D * D; x += kEncThreads)
            if (x / D != x % D) {
                const float y = G[(x / D) * L::kLd + x % D];
                off += y * y;
            }
        for (int o = 16; o; o >>= 1) off += __shfl_xor_sync(0xffffffffu, off, o);
        if ((tid & 31) == 0) red[tid >> 5] = off;
        __syncthreads();
        off = 0.f;
        for (int w = 0; w < kEncThreads / 32; ++w) off += red[w];
        __syncthreads();
        if (!(off > kJacobiTol * kJacobiTol * total)) break;  // (also ends on a zero G)
        for (int r = 0; r < D - 1; ++r) {
            if (tid < D / 2) {
                int pp, qq;
                pair_of(D, r, tid, pp, qq);
                const float gpp = G[pp * L::kLd + pp], gqq = G[qq * L::kLd + qq], gpq = G[pp * L::kLd + qq];
                float c = 1.f, s = 0.f;
                if (gpq != 0.f) {
                    // rotation that zeroes G[p][q]: t = tan(angle), the root of
                    // t^2 + 2 tau t - 1 = 0 of smaller magnitude
                    // (correctly rounded division and square root: with an
                    // approximate reciprocal square root the rotations are off
                    // orthogonal by a biased amount, which adds up over the
                    // sweeps and shrinks every eigenvalue)
                    const float tau = (gqq - gpp) / (2.f * gpq);
                    const float tt = copysignf(1.f, tau) / (fabsf(tau) + sqrtf(1.f + tau * tau));
                    c = 1.f / sqrtf(1.f + tt * tt);
                    s = tt * c;
                }
                rot[tid] = make_float4(c, s, __int_as_float(pp), __int_as_float(qq));
            }
            __syncthreads();
            // rows p, q of G: G <- R^T G (unrolled: the updates are
            // independent, so their shared-memory round trips overlap)
#pragma unroll 8
            for (int x = tid; x < (D / 2) * D; x += kEncThreads) {
                const float4 rr = rot[x / D];
                const int col = x % D, pp = __float_as_int(rr.z), qq = __float_as_int(rr.w);
                const float a = G[pp * L::kLd + col], bq = G[qq * L::kLd + col];
                G[pp * L::kLd + col] = rr.x * a - rr.y * bq;
                G[qq * L::kLd + col] = rr.y * a + rr.x * bq;
            }
            __syncthreads();
            // columns p, q of G and of V: G <- G R, V <- V R
#pragma unroll 8
            for (int x = tid; x < (D / 2) * D; x += kEncThreads) {
                const float4 rr = rot[x / D];
                const int row = x % D, pp = __float_as_int(rr.z), qq = __float_as_int(rr.w);
                const float a = G[row * L::kLd + pp], bq = G[row * L::kLd + qq];
                G[row * L::kLd + pp] = rr.x * a - rr.y * bq;
                G[row * L::kLd + qq] = rr.y * a + rr.x * bq;
                const float va = V[row * L::kLd + pp], vb = V[row * L::kLd + qq];
                V[row * L::kLd + pp] = rr.x * va - rr.y * vb;
                V[row * L::kLd + qq] = rr.y * va + rr.x * vb;
            }
            __syncthreads();
        }
    }
    // ---- eigenvalues: the Rayleigh quotients lambda_i = v_i^T G0 v_i / v_i^T v_i
    // of the accumulated rotation columns against the original G (the
    // rotated diagonal carries the rounding of every rotation, ~1e-5 of the
    // largest eigenvalue; the quotient ~1e-7), in a fixed summation order
    int *order = reinterpret_cast<int *>(X);  // [D]: position -> eigen index
    float *nrm = X + D;                       // [D]: v_i^T v_i
    float *lam = X + 2 * D;                   // [D]
    float *part = X + 3 * D;                  // [16][D]: partial quotients by row tile
    for (int i = tid; i < D; i += kEncThreads) {
        float nn = 0.f;
        for (int r = 0; r < D; ++r) nn = fmaf(V[r * L::kLd + i], V[r * L::kLd + i], nn);
        nrm[i] = nn;
    }
    {
        // thread (ti, tj): W[a][i] = sum_b G0[a][b] V[b][i] for its T x T tile,
        // then sum_a V[a][i] W[a][i] over its rows
        float w[T][T];
#pragma unroll
        for (int a = 0; a < T; ++a)
#pragma unroll
            for (int c = 0; c < T; ++c) w[a][c] = 0.f;
        for (int bb = 0; bb < D; ++bb) {
            float ga[T], vb[T];
#pragma unroll
            for (int a = 0; a < T; ++a) {
                ga[a] = g0[(T * ti + a) * D + bb];
                vb[a] = V[bb * L::kLd + T * tj + a];
            }
#pragma unroll
            for (int a = 0; a < T; ++a)
#pragma unroll
                for (int c = 0; c < T; ++c) w[a][c] = fmaf(ga[a], vb[c], w[a][c]);
        }
#pragma unroll
        for (int c = 0; c < T; ++c) {
            float sacc = 0.f;
#pragma unroll
            for (int a = 0; a < T; ++a) sacc = fmaf(V[(T * ti + a) * L::kLd + T * tj + c], w[a][c], sacc);
            part[ti * D + T * tj + c] = sacc;
        }
    }
    __syncthreads();
    for (int i = tid; i < D; i += kEncThreads) {
        float q = 0.f;
        for (int t = 0; t < 16; ++t) q += part[t * D + i];
        lam[i] = q / nrm[i];
    }
    __syncthreads();
    // descending order, ties by index
    for (int i = tid; i < D; i += kEncThreads) {
        const float li = lam[i];
        int pos = 0;
        for (int j = 0; j < D; ++j) {
            const float lj = lam[j];
            pos += (lj > li) || (lj == li && j < i);
        }
        order[pos] = i;
    }
    __syncthreads();
    float *sg = p.sigma + (int64_t)m * D;
    float *vt = p.vt + (int64_t)m * D * D;  // (G0 is no longer read)
    for (int x = tid; x < D; x += kEncThreads) sg[x] = sqrtf(fmaxf(lam[order[x]], 0.f));
    for (int x = tid; x < D * D; x += kEncThreads) {
        const int j = x / D, c = x % D;  // row j of B^T = column order[j] of V, unit length
        const int i = order[j];
        vt[x] = V[c * L::kLd + i] / sqrtf(nrm[i]);
    }
}

// Number of candidates of group (g, side) with sigma above (or at least) a
// value, over every block's positions [r0, cap).
__device__ __forceinline__ void group_caps(const EncParams &p, int b, int &r0, int &cap)
{
    const int avail = min(p.blen[b], p.d);
    r0 = min(p.r_min, avail);
    cap = min(p.r_max, avail);
}

__global__ void __launch_bounds__(kEncThreads) allocate_kernel(const EncParams p)
{
    __shared__ long long scan[kEncThreads];
    __shared__ long long s_ll[kEncThreads / 32];
    const int tid = threadIdx.x;
    const int g = blockIdx.x >> 1, side = blockIdx.x & 1;
    int32_t *rank = side ? p.rank_v : p.rank_k;
    const int64_t budget = side ? p.budget_v : p.budget_k;
    // the starting ranks and the number of units left to give
    long long used = 0, ncand = 0;
    for (int b = tid; b < p.nb; b += kEncThreads) {
        int r0, cap;
        group_caps(p, b, r0, cap);
        used += r0;
        ncand += max(0, cap - r0);
    }
    auto block_sum = [&](long long x) {
        for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
        __syncthreads();
        if ((tid & 31) == 0) s_ll[tid >> 5] = x;
        __syncthreads();
        long long t = 0;
        for (int w = 0; w < kEncThreads / 32; ++w) t += s_ll[w];
        return t;
    };
    used = block_sum(used);
    ncand = block_sum(ncand);
    const long long U = llmin(llmax(budget - used, 0), ncand);
    if (budget < used) {
        if (tid == 0) atomicCAS(p.status, 0, (int32_t)MILO_ERR_INVALID_ARG);
        return;
    }
    // candidates above a value (bits of a non-negative float order like the
    // value), over the flattened (block, j) space so that the loads are
    // independent and coalesced
    auto count_above = [&](uint32_t bits, bool or_equal) {
        long long c = 0;
        for (int64_t x = tid; x < (int64_t)p.nb * p.d; x += kEncThreads) {
            const int b = (int)(x / p.d), j = (int)(x % p.d);
            int r0, cap;
            group_caps(p, b, r0, cap);
            if (j < r0 || j >= cap) continue;
            const uint32_t u = __float_as_uint(p.sigma[(int64_t)(2 * (b * p.hkv + g) + side) * p.d + j]);
            c += or_equal ? (u >= bits) : (u > bits);
        }
        return block_sum(c);
    };
    // tau: the largest bits value with at least U candidates at or above it
    uint32_t tau = 0u;
    if (U > 0) {
        uint32_t lo = 0u, hi = 0x7f800000u;  // count(>= lo) >= U; search the largest such bits
        while (lo < hi) {
            const uint32_t mid = lo + (hi - lo + 1) / 2;
            if (count_above(mid, true) >= U) lo = mid; else hi = mid - 1;
        }
        tau = lo;
    }
    const long long above = U > 0 ? count_above(tau, false) : 0;
    long long need = U - above;  // candidates equal to tau to take, in (block, j) order
    // ranks: r0 + candidates above tau + the first `need` ties in order
    for (int b0 = 0; b0 < p.nb; b0 += kEncThreads) {
        const int b = b0 + tid;
        int take = 0, ties = 0;
        if (b < p.nb) {
            int r0, cap;
            group_caps(p, b, r0, cap);
            const float *sg = p.sigma + (int64_t)(2 * (b * p.hkv + g) + side) * p.d;
            for (int j = r0; j < cap && U > 0; ++j) {
                const uint32_t u = __float_as_uint(sg[j]);
                take += u > tau;
                ties += u == tau;
            }
            take += r0;
        }
        // exclusive scan of the ties over the blocks of this round
        scan[tid] = ties;
        __syncthreads();
        for (int o = 1; o < kEncThreads; o <<= 1) {
            const long long x = tid >= o ? scan[tid - o] : 0;
            __syncthreads();
            scan[tid] += x;
            __syncthreads();
        }
        const long long before = scan[tid] - ties;
        const long long total_ties = scan[kEncThreads - 1];
        __syncthreads();
        if (b < p.nb) {
            const long long mine = llmin(llmax(need - before, 0), ties);
            rank[b * p.hkv + g] = take + (int)mine;
        }
        need -= llmin(need, total_ties);
    }
}

template <int D>
__global__ void __launch_bounds__(kEncThreads) factor_kernel(const EncParams p)
{
    extern __shared__ __align__(16) uint8_t smem[];
    float *Vt = reinterpret_cast<float *>(smem);                 // [r][D + 1]
    float *X = Vt + D * (D + 1);                                  // [kEncTok][D + 1]
    const int tid = threadIdx.x;
    const int m = blockIdx.x, e = m >> 1, side = m & 1;
    const int b = e / p.hkv, g = e % p.hkv;
    const int n = p.blen[b];
    // (the ranks are at most the region's capacity, min(r_max, n, d): clamp
    // them anyway, so that a bad rank array cannot write past the region)
    const int r = max(0, min(side ? p.rank_v[e] : p.rank_k[e], min(p.r_max, min(n, D))));
    const uint16_t *src = (side ? p.v : p.k) + (p.tok0[b] * p.hkv + g) * (int64_t)D;
    const int64_t rstride = (int64_t)p.hkv * D;
    const float *vt = p.vt + (int64_t)m * D * D;
    uint16_t *C = p.arena + p.offs[(int64_t)e * 4 + (side ? 2 : 0)];
    uint16_t *P = p.arena + p.offs[(int64_t)e * 4 + (side ? 3 : 1)];
    if (r == 0) return;
    for (int x = tid; x < r * D; x += kEncThreads) {
        const float y = vt[x];
        Vt[(x / D) * (D + 1) + x % D] = y;
        const __nv_bfloat16 h = __float2bfloat16_rn(y);
        P[x] = *reinterpret_cast<const uint16_t *>(&h);
    }
    // thread (tt, jj): tokens 4 tt .. 4 tt + 3 of a tile, columns RJ jj .. of C
    constexpr int RJ = D / 16;
    const int tt = tid / 16, jj = tid % 16;
    for (int t0 = 0; t0 < n; t0 += kEncTok) {
        const int nt = min(kEncTok, n - t0);
        __syncthreads();
        for (int x = tid; x < kEncTok * D; x += kEncThreads) {
            const int t = x / D, c = x % D;
            X[t * (D + 1) + c] = t < nt ? bf16f(src[(int64_t)(t0 + t) * rstride + c]) : 0.f;
        }
        __syncthreads();
        // C[t][j] = sum_c X[t][c] Vt[j][c]
        if (RJ * jj < r && 4 * tt < nt) {
            float acc[4][RJ];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int c = 0; c < RJ; ++c) acc[a][c] = 0.f;
#pragma unroll 4
            for (int c = 0; c < D; ++c) {
                float xa[4], vb[RJ];
#pragma unroll
                for (int a = 0; a < 4; ++a) xa[a] = X[(4 * tt + a) * (D + 1) + c];
#pragma unroll
                for (int q = 0; q < RJ; ++q) vb[q] = Vt[(RJ * jj + q) * (D + 1) + c];
#pragma unroll
                for (int a = 0; a < 4; ++a)
#pragma unroll
                    for (int q = 0; q < RJ; ++q) acc[a][q] = fmaf(xa[a], vb[q], acc[a][q]);
            }
#pragma unroll
            for (int a = 0; a < 4; ++a) {
                const int t = 4 * tt + a;
                if (t >= nt) continue;
#pragma unroll
                for (int q = 0; q < RJ; ++q) {
                    const int j = RJ * jj + q;
                    if (j >= r) continue;
                    const __nv_bfloat16 h = __float2bfloat16_rn(acc[a][q]);
                    C[(int64_t)(t0 + t) * r + j] = *reinterpret_cast<const uint16_t *>(&h);
                }
            }
        }
    }
}

template <class K>
cudaError_t set_smem(K kernel, int bytes)
{
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

}  // namespace

int64_t encode_layout(int nb, int hkv, int d, const int32_t *blen, int r_max, int64_t *offs)
{
    int64_t cur = 0;
    for (int b = 0; b < nb; ++b)
        for (int g = 0; g < hkv; ++g) {
            const int64_t e = (int64_t)b * hkv + g;
            const int n = blen[b];
            const int cap = std::min(std::min(r_max, n), d);
            const int64_t sz[4] = {(int64_t)n * cap, (int64_t)cap * d, (int64_t)n * cap, (int64_t)cap * d};
            for (int f = 0; f < 4; ++f) {
                if (offs) offs[e * 4 + f] = cur;
                cur += (sz[f] + 7) / 8 * 8;
            }
        }
    return cur;
}

cudaError_t launch_encode(const uint16_t *k, const uint16_t *v, const int64_t *tok0, const int32_t *blen,
                          const int64_t *offs, uint16_t *arena, int32_t *rank_k, int32_t *rank_v, float *sigma,
                          float *vt, int32_t *status, int nb, int hkv, int d, int r_min, int r_max,
                          int64_t budget_k, int64_t budget_v, cudaStream_t stream)
{
    EncParams p{k, v, tok0, blen, offs, arena, rank_k, rank_v, sigma, vt, status, nb, hkv, d, r_min, r_max,
                budget_k, budget_v};
    const int mats = 2 * nb * hkv;
    cudaError_t e;
    if (d == 64) {
        if ((e = set_smem(spectrum_kernel<64>, EncLay<64>::kTotal)) != cudaSuccess) return e;
        spectrum_kernel<64><<<mats, kEncThreads, EncLay<64>::kTotal, stream>>>(p);
    } else {
        if ((e = set_smem(spectrum_kernel<128>, EncLay<128>::kTotal)) != cudaSuccess) return e;
        spectrum_kernel<128><<<mats, kEncThreads, EncLay<128>::kTotal, stream>>>(p);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    allocate_kernel<<<2 * hkv, kEncThreads, 0, stream>>>(p);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int fsmem = (d * (d + 1) + kEncTok * (d + 1)) * 4;
    if (d == 64) {
        if ((e = set_smem(factor_kernel<64>, fsmem)) != cudaSuccess) return e;
        factor_kernel<64><<<mats, kEncThreads, fsmem, stream>>>(p);
    } else {
        if ((e = set_smem(factor_kernel<128>, fsmem)) != cudaSuccess) return e;
        factor_kernel<128><<<mats, kEncThreads, fsmem, stream>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace milo
