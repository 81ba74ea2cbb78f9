// milo_merge.cuh -- the shared-reference merge of the split softmax, used by
// every item of a decode call: the chunk grid's prefix chunks and dense-tail
// items and the tensor-core grid's runs.
//
// Every item ends with (o, m, l) per query row: o = sum 2^(s - m) v over its
// tokens, l = sum 2^(s - m) (Eq. 1 on a partition of the tokens).  Rather
// than storing these and merging them afterwards, each item adds 2^(m - M) o
// and 2^(m - M) l into fp32 accumulators of its KV head with vector
// reductions, for one reference M per row: the first item to finish a tile
// sets M = its running maximum + kRefMargin (compare-and-swap), and every
// other item reads it back.  With M within kDirectMax below an item's maximum
// nothing overflows; an item whose maximum lies further above M (a rare
// outlier) writes its record instead and lists it.  Once the grid is done,
// the finish grid divides the accumulators by the sum, folds in the listed
// records by the log-sum-exp rule, writes the output and clears the
// accumulators for the next call.
#pragma once
#include <cstdint>

#include "milo_internal.h"

namespace milo {
namespace {

constexpr float kRefMargin = 40.f;  // M = first tile maximum + this
constexpr float kDirectMax = 60.f;  // items with m - M above this keep a record

// A reference maximum is stored as its float bits with the sign flipped, so
// that 0 means "not set" (x + kRefMargin is never -0).
__device__ __forceinline__ uint32_t ref_enc(float x) { return __float_as_uint(x) ^ 0x80000000u; }
__device__ __forceinline__ float ref_dec(uint32_t u) { return __uint_as_float(u ^ 0x80000000u); }

// Lane c4 == 0 of each valid row sets or reads the row's reference; the
// result arrives later (it is used only at the end of the item).
__device__ __forceinline__ uint32_t publish_ref(const DecodeParams &p, int g, int arow, bool row_ok, int c4, float m)
{
    uint32_t got = 0u;
    if (c4 == 0 && row_ok) {
        const uint32_t mine = ref_enc(m + kRefMargin);
        const uint32_t old = atomicCAS(p.acc_m + (int64_t)g * p.rows_max + arow, 0u, mine);
        got = old ? old : mine;
    }
    return got;
}

}  // namespace
}  // namespace milo
