// milo_pack.cu -- copy a layer's low-rank factors (the paper's low-rank cache,
// Alg. 1 Stage 1 "LC.Store") from the logical row-major layout of the block
// table into the packed layout the decode kernel streams:
//   * ranks zero-padded to a multiple of 8, coefficient tokens to a multiple
//     of 8;
//   * 8x8 bf16 cores of 128 contiguous bytes (each core row is one 16-byte
//     line): for C, [token group][rank group] over the whole entry, so a 1-D
//     bulk copy of any token range lands in shared memory as evenly strided
//     cores (what ldmatrix and tensor-core shared-memory descriptors read).
// The copy is bit-exact; padding is zero, so NaN-filled gaps between the
// caller's factors never reach the packed arena.
#include <cuda_bf16.h>

#include "milo_internal.h"

namespace milo {
namespace {

__global__ void __launch_bounds__(256) pack_kernel(const uint16_t *__restrict__ arena,
                                                   const EntryDev *__restrict__ entries,
                                                   const int64_t *__restrict__ loff,
                                                   int head_dim, uint8_t *__restrict__ packed)
{
    const int e = blockIdx.x, f = blockIdx.y;  // f: 0 C^K, 1 P^K, 2 C^V, 3 P^V
    const EntryDev ent = entries[e];
    const int r = (f < 2) ? ent.rk : ent.rv;
    const int r8 = (r + 7) & ~7;
    const int64_t src0 = loff[4 * e + f];
    const int64_t dst0 = (f == 0) ? ent.off_ck : (f == 1) ? ent.off_pk : (f == 2) ? ent.off_cv : ent.off_pv;
    const uint16_t *src = arena + src0;
    uint8_t *dst = packed + dst0;
    if (r8 == 0) return;
    if ((f & 1) == 0) {
        // coefficients C (n x r): 8x8 cores [token group][rank group] over the whole
        // entry, so token groups are evenly spaced (r8/8 cores apart)
        const int n = ent.n, n8 = (n + 7) & ~7, nrg = r8 / 8;
        const int64_t chunks = (int64_t)n8 * r8 / 8;
        for (int64_t qi = threadIdx.x; qi < chunks; qi += blockDim.x) {
            const int core = (int)(qi / 8), row = (int)(qi % 8);
            const int tg = core / nrg, rg = core % nrg;
            const int t = 8 * tg + row;
            const int j0 = 8 * rg;
            alignas(16) uint16_t v[8];
#pragma unroll
            for (int x = 0; x < 8; ++x) {
                const int j = j0 + x;
                v[x] = (t < n && j < r) ? src[(int64_t)t * r + j] : (uint16_t)0;
            }
            *reinterpret_cast<uint4 *>(dst + qi * 16) = *reinterpret_cast<const uint4 *>(v);
        }
    } else {
        // basis P (r x d): [rank group][column group]
        const int cgs = head_dim / 8;
        const int chunks = r8 * cgs;
        for (int qi = threadIdx.x; qi < chunks; qi += blockDim.x) {
            const int core = qi / 8, row = qi % 8;
            const int jg = core / cgs, cg = core % cgs;
            const int j = 8 * jg + row;
            alignas(16) uint16_t v[8];
#pragma unroll
            for (int x = 0; x < 8; ++x)
                v[x] = (j < r) ? src[(int64_t)j * head_dim + 8 * cg + x] : (uint16_t)0;
            *reinterpret_cast<uint4 *>(dst + (int64_t)qi * 16) = *reinterpret_cast<const uint4 *>(v);
        }
    }
}

}  // namespace

cudaError_t launch_pack(const void *arena, const EntryDev *entries_dev,
                        const int64_t *logical_offsets_dev, int num_entries,
                        int head_dim, uint8_t *packed, int64_t packed_bytes,
                        cudaStream_t stream)
{
    if (num_entries == 0) return cudaSuccess;
    cudaError_t err = cudaMemsetAsync(packed, 0, (size_t)packed_bytes, stream);
    if (err != cudaSuccess) return err;
    dim3 grid(num_entries, 4);
    pack_kernel<<<grid, 256, 0, stream>>>(static_cast<const uint16_t *>(arena), entries_dev,
                                          logical_offsets_dev, head_dim, packed);
    return cudaGetLastError();
}

}  // namespace milo
