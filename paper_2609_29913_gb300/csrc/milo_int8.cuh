// milo_int8.cuh -- the read-back of one row of an INT8 core (the group-wise
// asymmetric INT8 storage of Sec. 5.3, Table 2), shared by the staging
// kernels and the chunk grid's direct reads, so that both give the same
// bf16 values bit for bit.
#pragma once
#include <cstdint>

#include <cuda_bf16.h>

namespace milo {
namespace {

// Packed fp32 pairs (x in the low half of a 64-bit register pair); each lane
// of the paired subtract and fused multiply-add rounds as the scalar
// instruction does.
__device__ __forceinline__ uint64_t pair(uint32_t x, uint32_t y)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(x), "r"(y));
    return r;
}
__device__ __forceinline__ uint32_t bf16x2_of(uint64_t v)
{
    float x, y;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(v));
    __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
    return *reinterpret_cast<uint32_t *>(&h);
}

// One 8-value row of a core: codes c (bytes in element order) and the group's
// parameter word -> 8 bf16 values bf16(m + s c).  A code byte b becomes the
// float 2^23 + b by placing it under the exponent of 2^23 (exact), then
// 2^23 is subtracted (exact) and m + s b is one fused multiply-add (s b is
// exact: s has 8 significant bits, b at most 8), as in the scalar form.
__device__ __forceinline__ uint4 dequant_row(uint2 c, uint32_t pw)
{
    const uint32_t mb = pw << 16, sb = pw & 0xFFFF0000u;
    const uint64_t m2 = pair(mb, mb), s2 = pair(sb, sb), k2 = pair(0x4B000000u, 0x4B000000u);
    uint32_t out[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t word = (i < 2) ? c.x : c.y;
        const uint32_t b0 = 2 * (i & 1);
        uint64_t v = pair(__byte_perm(word, 0x4B000000u, 0x7540u | b0), __byte_perm(word, 0x4B000000u, 0x7540u | (b0 + 1)));
        asm("sub.rn.f32x2 %0, %0, %1;" : "+l"(v) : "l"(k2));
        asm("fma.rn.f32x2 %0, %1, %0, %2;" : "+l"(v) : "l"(s2), "l"(m2));
        out[i] = bf16x2_of(v);
    }
    return make_uint4(out[0], out[1], out[2], out[3]);
}

}  // namespace
}  // namespace milo
