// milo_host.cpp -- host side of the libmilo C ABI (include/milo.h):
// table validation, packed layout, static work partition, plan lifecycle and
// the decode launch.  No exception crosses the ABI.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "milo.h"
#include "milo_internal.h"

using namespace milo;

namespace {

thread_local std::string g_last_error;

milo_status_t cuda_fail(cudaError_t e, const char *what)
{
    g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
    return MILO_ERR_CUDA;
}

milo_status_t fail(milo_status_t s, const std::string &msg)
{
    g_last_error = msg;
    return s;
}

inline int r8(int r) { return (r + 7) & ~7; }
inline int64_t align_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

struct Seg {
    int32_t entry, t0, t1, slot, flags;
};

milo_status_t validate(const milo_block_table_t *t)
{
    if (!t) return fail(MILO_ERR_INVALID_ARG, "table is null");
    if (t->num_blocks < 0 || t->num_kv_heads < 1)
        return fail(MILO_ERR_INVALID_ARG, "num_blocks < 0 or num_kv_heads < 1");
    if (t->head_dim != 64 && t->head_dim != 128)
        return fail(MILO_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (t->num_blocks == 0) return MILO_OK;
    if (!t->block_len || !t->rank_k || !t->rank_v || !t->off_ck || !t->off_pk || !t->off_cv || !t->off_pv)
        return fail(MILO_ERR_INVALID_ARG, "null table array");
    if (t->arena_elems < 0) return fail(MILO_ERR_INVALID_ARG, "arena_elems < 0");
    if (t->arena_elems > 0 && !t->arena) return fail(MILO_ERR_INVALID_ARG, "arena is null");
    if (reinterpret_cast<uintptr_t>(t->arena) % 16 != 0)
        return fail(MILO_ERR_ALIGNMENT, "arena is not 16-byte aligned");
    const int d = t->head_dim, H = t->num_kv_heads;
    struct Region { int64_t a, b; };
    std::vector<Region> regions;
    regions.reserve((size_t)t->num_blocks * H * 4);
    for (int b = 0; b < t->num_blocks; ++b) {
        const int n = t->block_len[b];
        if (n < 1 || n > 65536) return fail(MILO_ERR_BAD_TABLE, "block length outside [1, 65536]");
        for (int g = 0; g < H; ++g) {
            const int64_t e = (int64_t)b * H + g;
            const int rk = t->rank_k[e], rv = t->rank_v[e];
            if (rk < 0 || rk > d || rv < 0 || rv > d) return fail(MILO_ERR_BAD_TABLE, "rank outside [0, head_dim]");
            const int64_t off[4] = {t->off_ck[e], t->off_pk[e], t->off_cv[e], t->off_pv[e]};
            const int64_t sz[4] = {(int64_t)n * rk, (int64_t)rk * d, (int64_t)n * rv, (int64_t)rv * d};
            for (int f = 0; f < 4; ++f) {
                if (off[f] % 8 != 0) return fail(MILO_ERR_ALIGNMENT, "factor offset not a multiple of 8 elements");
                if (off[f] < 0 || off[f] + sz[f] > t->arena_elems)
                    return fail(MILO_ERR_BAD_TABLE, "factor region outside the arena");
                if (sz[f] > 0) regions.push_back({off[f], off[f] + sz[f]});
            }
        }
    }
    std::sort(regions.begin(), regions.end(), [](const Region &x, const Region &y) { return x.a < y.a; });
    for (size_t i = 1; i < regions.size(); ++i)
        if (regions[i].a < regions[i - 1].b) return fail(MILO_ERR_BAD_TABLE, "factor regions overlap");
    return MILO_OK;
}

// Packed byte offsets [E][4] (C^K, P^K, C^V, P^V), each 128-byte aligned.
int64_t packed_layout(const milo_block_table_t *t, std::vector<int64_t> &offs)
{
    const int H = t->num_kv_heads, d = t->head_dim;
    const int64_t E = (int64_t)t->num_blocks * H;
    offs.assign((size_t)E * 4, 0);
    int64_t cur = 0;
    for (int64_t e = 0; e < E; ++e) {
        const int n8 = (t->block_len[e / H] + 7) & ~7;
        const int64_t sz[4] = {(int64_t)n8 * r8(t->rank_k[e]) * 2, (int64_t)r8(t->rank_k[e]) * d * 2,
                               (int64_t)n8 * r8(t->rank_v[e]) * 2, (int64_t)r8(t->rank_v[e]) * d * 2};
        for (int f = 0; f < 4; ++f) {
            offs[(size_t)e * 4 + f] = cur;
            cur = align_up(cur + sz[f], 128);
        }
    }
    return cur;
}

// Cost of the tensor-core decode's work, in eighths of a cycle of one SM: per
// token the softmax of a 128-row tile (~8 cycles) and the hi + lo score and
// value products (ranks rounded up to 16: (r^k + r^v) / 8 cycles); per
// segment the projection, the staging of q~ and v~ and the back-projection
// (~7500 cycles), charged with its first tile.  (A segment weight of 2500,
// 5000, 7500 and 10000 cycles measured 0.433, 0.429, 0.425 and 0.428 ms on
// the 1M-token layer and 3.37, 3.31, 3.27 and 3.27 ms on the batch-64 step.)
struct TensorCost {
    const milo_block_table_t *t;
    static int r16(int r) { return (r + 15) & ~15; }
    int64_t tile(int e, int t8) const { return (int64_t)t8 * (64 + r16(t->rank_k[e]) + r16(t->rank_v[e])); }
    int64_t first(int) const { return 60000; }
    int64_t last(int) const { return 0; }
};
constexpr int64_t kTcMinShareCost = 100000;  // in TensorCost units: ~one 512-token entry of rank 64

// Static partition of the prefix over `P` shares of the tensor-core grid,
// under a cost model: segments (entry, token range) listed share by share
// (share c holds segs[cta_begin[c] .. cta_begin[c + 1])), each share's
// segments grouped in runs of one KV head, one accumulator slot per run.
template <class Cost>
void partition_with(const milo_block_table_t *t, int P, const Cost &cost, std::vector<Seg> &segs,
                    std::vector<int32_t> &cta_begin, int &num_slots)
{
    const int H = t->num_kv_heads, nb = t->num_blocks;
    int64_t total = 0;
    for (int g = 0; g < H; ++g)
        for (int b = 0; b < nb; ++b) {
            const int e = b * H + g, n = t->block_len[b];
            total += cost.first(e) + cost.last(e);
            for (int t0 = 0; t0 < n; t0 += kTileTokens) total += cost.tile(e, (std::min(n - t0, kTileTokens) + 7) & ~7);
        }
    segs.clear();
    cta_begin.assign((size_t)P + 1, 0);
    // Cost line: entries (KV-head-major, then block order), each charged its
    // 32-token tiles, with the entry's first and last charges on its first and
    // last tile.  A tile belongs to the share (c total/P, (c+1) total/P] that
    // contains the midpoint of the tile's cost interval.  A block cut between
    // two shares is read again for its bases by the second (from L2).
    int cta = 0;
    int64_t pos = 0;
    for (int g = 0; g < H; ++g)
        for (int b = 0; b < nb; ++b) {
            const int e = b * H + g, n = t->block_len[b];
            bool open = false;
            for (int t0 = 0; t0 < n; t0 += kTileTokens) {
                const int t1 = std::min(n, t0 + kTileTokens);
                const int64_t c = cost.tile(e, (t1 - t0 + 7) & ~7) + (t0 == 0 ? cost.first(e) : 0) +
                                  (t1 == n ? cost.last(e) : 0);
                const double mid = (double)pos + 0.5 * (double)c;
                int owner = total > 0 ? (int)(mid * P / (double)total) : 0;
                owner = std::min(std::max(owner, cta), P - 1);
                if (owner != cta) {
                    for (int x = cta + 1; x <= owner; ++x) cta_begin[x] = (int32_t)segs.size();
                    cta = owner;
                    open = false;
                }
                if (!open) {
                    segs.push_back({e, t0, t0, 0, 0});
                    open = true;
                }
                segs.back().t1 = t1;
                pos += c;
            }
        }
    for (int c = cta + 1; c <= P; ++c) cta_begin[c] = (int32_t)segs.size();
    // runs and slots: consecutive segments of one share with one KV head
    num_slots = 0;
    for (int c = 0; c < P; ++c) {
        int prev_g = -1;
        for (int s = cta_begin[c]; s < cta_begin[c + 1]; ++s) {
            const int g = segs[s].entry % H;
            if (g != prev_g) {
                segs[s].flags |= kSegFirstOfRun;
                if (s > cta_begin[c]) segs[s - 1].flags |= kSegLastOfRun;
                ++num_slots;
                prev_g = g;
            }
            segs[s].slot = num_slots - 1;
        }
        if (cta_begin[c + 1] > cta_begin[c]) segs[cta_begin[c + 1] - 1].flags |= kSegLastOfRun;
    }
}


// Chunks of the chunk grid: every prefix entry, KV-head-major then in
// block order, cut into the fewest token ranges of at most kChunkMaxTok tokens
// whose coefficient rows (C^K and C^V, rounded up to 8 tokens) fit
// kChunkBytes, of about equal length; a range starts at a multiple of 32
// tokens.  f(entry, KV head, t0, t1) for each range in that order.
template <class F>
void for_each_chunk(const milo_block_table_t *t, F &&f)
{
    const int H = t->num_kv_heads, nb = t->num_blocks;
    for (int g = 0; g < H; ++g) {
        for (int b = 0; b < nb; ++b) {
            const int e = b * H + g, n = t->block_len[b];
            const int rk8 = r8(t->rank_k[e]), rv8 = r8(t->rank_v[e]);
            // the fewest chunks within the byte budget, then equal token
            // ranges (multiples of 32), so that an entry's chunks take
            // about equally long
            // (an entry of rank 0 in K and V has no coefficient rows: its
            // tokens go in 32-token ranges, whose pieces copy nothing)
            const int row_bytes = (rk8 + rv8) * 2;
            const int most = row_bytes > 0 ? std::max(32, std::min(kChunkMaxTok, kChunkBytes / row_bytes / 32 * 32))
                                           : 32;
            const int nch = std::max(1, (n + most - 1) / most);
            const int tok = ((n + nch - 1) / nch + 31) / 32 * 32;
            for (int t0 = 0; t0 < n; t0 += tok) f(e, g, t0, std::min(n, t0 + tok));
        }
    }
}

void build_chunks(const milo_block_table_t *t, const std::vector<int64_t> &poffs, std::vector<ChunkDev> &chunks,
                  std::vector<int32_t> &g_begin)
{
    const int H = t->num_kv_heads;
    chunks.clear();
    g_begin.assign((size_t)H + 1, 0);
    for_each_chunk(t, [&](int e, int g, int t0, int t1) {
        const int n = t->block_len[e / H];
        const int rk8 = r8(t->rank_k[e]), rv8 = r8(t->rank_v[e]), n8 = r8(n);
        ChunkDev c = {};
        c.ck = poffs[(size_t)e * 4 + 0] + (int64_t)t0 * rk8 * 2;
        c.pk = poffs[(size_t)e * 4 + 1];
        c.cv = poffs[(size_t)e * 4 + 2] + (int64_t)t0 * rv8 * 2;
        c.pv = poffs[(size_t)e * 4 + 3];
        c.ntok = t1 - t0;
        c.tok8 = std::min(r8(t1), n8) - t0;
        c.nrk = rk8 / 8;
        c.nrv = rv8 / 8;
        c.g = g;
        c.rk = t->rank_k[e];
        c.rv = t->rank_v[e];
        chunks.push_back(c);
        g_begin[(size_t)g + 1] = (int32_t)chunks.size();
    });
    // a KV head without chunks starts where the previous one ended
    for (int g = 1; g <= H; ++g) g_begin[(size_t)g] = std::max(g_begin[(size_t)g], g_begin[(size_t)g - 1]);
}

// The plan's accumulator buffer: the reference maxima [H][R] (R = 8 x the
// row groups of 8 rows), the list counts [H][R / 8], and at a 16-byte
// boundary the row sums [H][R] and the output accumulators [H][R][d].
size_t acc_l_offset(int H, int R)
{
    return (sizeof(uint32_t) * (size_t)H * (R + R / 8) + 15) / 16 * 16;
}
size_t acc_bytes(int H, int R, int d)
{
    return acc_l_offset(H, R) + sizeof(float) * (size_t)H * R * (1 + (size_t)d);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

}  // namespace

struct milo_prefix {
    int device = 0;
    int nb = 0, hkv = 0, hq = 0, d = 0, G = 0, max_batch = 0;
    int max_nrg = 0;
    int64_t prefix_tokens = 0, logical_bytes = 0, packed_bytes = 0;
    uint8_t *packed = nullptr;        // the arena the kernels read (an offloaded plan: the staged copy)
    uint8_t *packed_host = nullptr;   // offloaded plans: the arena in pinned host memory
    // INT8 plans (milo_prefix_quantize_int8): codes then parameters in one
    // allocation, device memory or mapped pinned host memory
    uint8_t *int8_store = nullptr;    // the allocation (cudaFree / cudaFreeHost)
    const uint8_t *int8_dev = nullptr;  // its address as the kernels see it
    bool int8_host = false;
    int64_t max_factor_groups = 0;    // the most 8x8 cores of one factor
    EntryDev *entries = nullptr;
    ChunkDev *chunks = nullptr;       // the chunk grid's prefix chunks, KV-head-major
    int num_chunks = 0;
    int max_head_chunks = 0;          // the most chunks of one KV head
    uint8_t *acc = nullptr;            // the chunk grid's per-row accumulators (zero between calls)
    int32_t *status = nullptr;
    // tensor-core path: one partition per share count a call can use
    bool tc = false;                  // the tensor-core partitions exist (a plan with a prefix)
    int tc_min_rows = kTcMinRows;     // calls with at least this many rows per KV head take them
    struct TcPart {
        int nshare, seg0, num_slots, max_runs;  // segments at tc_segs + seg0, shares at tc_cta + cta0
        int cta0;
    };
    std::vector<TcPart> tc_parts;
    TcSegDev *tc_segs = nullptr;
    int32_t *tc_cta = nullptr;
    int sms = 0;
    int tc_max_shares = 0;            // shares worth at least kTcMinShareCost each
    // reconstruct-then-attend: chunks of at most kRcChunkTiles tiles of one entry
    int4 *rc_chunks = nullptr;
    int rc_num_chunks = 0, rc_max_head_chunks = 0;
    // pre-RoPE factors (milo_prefix_set_rope): rotation tables, or null
    float2 *rope_tile = nullptr, *rope_off = nullptr;
    int32_t *rope_tile_base = nullptr;
    int tc_shares(int64_t ntile) const
    {
        return (int)std::max<int64_t>(1, std::min<int64_t>(sms / std::max<int64_t>(1, ntile), tc_max_shares));
    }
    const TcPart *tc_part(int ntile) const
    {
        const int ns = tc_shares(ntile);
        for (const TcPart &t : tc_parts)
            if (t.nshare == ns) return &t;
        return nullptr;
    }
};

extern "C" {

const char *milo_status_string(int32_t s)
{
    switch (s) {
    case MILO_OK: return "ok";
    case MILO_ERR_INVALID_ARG: return "invalid argument";
    case MILO_ERR_BAD_TABLE: return "inconsistent block table";
    case MILO_ERR_ALIGNMENT: return "misaligned pointer or offset";
    case MILO_ERR_UNSUPPORTED: return "unsupported configuration";
    case MILO_ERR_CUDA: return "CUDA runtime error";
    case MILO_ERR_TIMEOUT: return "device wait timed out";
    case MILO_ERR_DEVICE_BOUNDS: return "device-side bounds check failed";
    case MILO_ERR_WORKSPACE: return "workspace missing or too small";
    default: return "unknown status";
    }
}

int32_t milo_version(void) { return 200; }

const char *milo_last_error_message(void) { return g_last_error.c_str(); }

milo_status_t milo_validate_table(const milo_block_table_t *table) { return validate(table); }

milo_status_t milo_packed_layout(const milo_block_table_t *table, int64_t *packed_offsets, int64_t *total_bytes)
{
    milo_status_t s = validate(table);
    if (s != MILO_OK) return s;
    std::vector<int64_t> offs;
    const int64_t total = packed_layout(table, offs);
    if (packed_offsets) std::memcpy(packed_offsets, offs.data(), offs.size() * sizeof(int64_t));
    if (total_bytes) *total_bytes = total;
    return MILO_OK;
}

milo_status_t milo_partition_prefix(const milo_block_table_t *table, int32_t num_shares, int32_t max_segments,
                                    int32_t *seg_entry, int32_t *seg_t0, int32_t *seg_t1, int32_t *seg_slot,
                                    int32_t *share_begin, int32_t *num_segments, int32_t *num_slots)
{
    milo_status_t s = validate(table);
    if (s != MILO_OK) return s;
    if (num_shares < 1) return fail(MILO_ERR_INVALID_ARG, "num_shares < 1");
    std::vector<Seg> segs;
    std::vector<int32_t> cb;
    int ns = 0;
    partition_with(table, num_shares, TensorCost{table}, segs, cb, ns);
    if (num_segments) *num_segments = (int32_t)segs.size();
    if (num_slots) *num_slots = ns;
    if (share_begin) std::memcpy(share_begin, cb.data(), cb.size() * sizeof(int32_t));
    if (seg_entry || seg_t0 || seg_t1 || seg_slot) {
        if ((int64_t)segs.size() > max_segments) return fail(MILO_ERR_INVALID_ARG, "max_segments too small");
        for (size_t i = 0; i < segs.size(); ++i) {
            if (seg_entry) seg_entry[i] = segs[i].entry;
            if (seg_t0) seg_t0[i] = segs[i].t0;
            if (seg_t1) seg_t1[i] = segs[i].t1;
            if (seg_slot) seg_slot[i] = segs[i].slot;
        }
    }
    return MILO_OK;
}

milo_status_t milo_chunk_prefix(const milo_block_table_t *table, int32_t max_chunks, int32_t *chunk_entry,
                                int32_t *chunk_t0, int32_t *chunk_t1, int32_t *num_chunks)
{
    milo_status_t s = validate(table);
    if (s != MILO_OK) return s;
    int32_t n = 0;
    const bool fill = chunk_entry || chunk_t0 || chunk_t1;
    bool overflow = false;
    for_each_chunk(table, [&](int e, int, int t0, int t1) {
        if (fill && n < max_chunks) {
            if (chunk_entry) chunk_entry[n] = e;
            if (chunk_t0) chunk_t0[n] = t0;
            if (chunk_t1) chunk_t1[n] = t1;
        } else if (fill) {
            overflow = true;
        }
        ++n;
    });
    if (num_chunks) *num_chunks = n;
    if (overflow) return fail(MILO_ERR_INVALID_ARG, "max_chunks too small");
    return MILO_OK;
}

milo_status_t milo_prefix_destroy(milo_prefix_t *plan)
{
    if (!plan) return MILO_OK;
    int cur = 0;
    cudaGetDevice(&cur);
    cudaSetDevice(plan->device);
    cudaDeviceSynchronize();
    // (a staged copy belongs to the caller)
    if (plan->packed_host) cudaFreeHost(plan->packed_host);
    else if (plan->int8_store) {
        if (plan->int8_host) cudaFreeHost(plan->int8_store);
        else cudaFree(plan->int8_store);
    } else cudaFree(plan->packed);
    cudaFree(plan->entries);
    cudaFree(plan->chunks);
    cudaFree(plan->acc);
    cudaFree(plan->status);
    cudaFree(plan->tc_segs);
    cudaFree(plan->tc_cta);
    cudaFree(plan->rc_chunks);
    cudaFree(plan->rope_tile);
    cudaFree(plan->rope_off);
    cudaFree(plan->rope_tile_base);
    cudaSetDevice(cur);
    delete plan;
    return MILO_OK;
}

milo_status_t milo_prefix_create(const milo_block_table_t *table, int32_t num_q_heads, int32_t max_batch,
                                 void *stream_, milo_prefix_t **out_plan)
{
    if (!out_plan) return fail(MILO_ERR_INVALID_ARG, "out_plan is null");
    *out_plan = nullptr;
    milo_status_t s = validate(table);
    if (s != MILO_OK) return s;
    if (num_q_heads < 1 || num_q_heads % table->num_kv_heads != 0)
        return fail(MILO_ERR_INVALID_ARG, "num_q_heads must be a positive multiple of num_kv_heads");
    if (max_batch < 1) return fail(MILO_ERR_INVALID_ARG, "max_batch < 1");
    const int G = num_q_heads / table->num_kv_heads;
    // query rows per KV head are counted in int on the device
    if ((int64_t)max_batch * G > (1 << 30)) return fail(MILO_ERR_UNSUPPORTED, "max_batch x G above 2^30");
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);

    milo_prefix *p = new (std::nothrow) milo_prefix;
    if (!p) return fail(MILO_ERR_INVALID_ARG, "out of host memory");
    cudaError_t e = cudaGetDevice(&p->device);
    if (e != cudaSuccess) { delete p; return cuda_fail(e, "cudaGetDevice"); }
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, p->device);
    if (e != cudaSuccess) { delete p; return cuda_fail(e, "cudaDeviceGetAttribute"); }
    const int H = table->num_kv_heads, d = table->head_dim, nb = table->num_blocks;
    p->nb = nb; p->hkv = H; p->hq = num_q_heads; p->d = d; p->G = G; p->max_batch = max_batch;
    p->max_nrg = (max_batch * G + 7) / 8;

    std::vector<int64_t> poffs;
    p->packed_bytes = packed_layout(table, poffs);

    const int64_t E = (int64_t)nb * H;
    std::vector<EntryDev> ents((size_t)E);
    std::vector<int64_t> loffs((size_t)E * 4);
    for (int64_t x = 0; x < E; ++x) {
        EntryDev &en = ents[(size_t)x];
        en.off_ck = poffs[(size_t)x * 4 + 0];
        en.off_pk = poffs[(size_t)x * 4 + 1];
        en.off_cv = poffs[(size_t)x * 4 + 2];
        en.off_pv = poffs[(size_t)x * 4 + 3];
        en.n = table->block_len[x / H];
        en.rk = table->rank_k[x];
        en.rv = table->rank_v[x];
        en.g = (int)(x % H);
        {   // the most 8x8 cores of one factor (the INT8 staging grid's extent)
            const int64_t n8 = (en.n + 7) / 8, d8 = table->head_dim / 8;
            const int64_t k8 = (en.rk + 7) / 8, v8 = (en.rv + 7) / 8;
            p->max_factor_groups = std::max({p->max_factor_groups, n8 * k8, n8 * v8, k8 * d8, v8 * d8});
        }
        loffs[(size_t)x * 4 + 0] = table->off_ck[x];
        loffs[(size_t)x * 4 + 1] = table->off_pk[x];
        loffs[(size_t)x * 4 + 2] = table->off_cv[x];
        loffs[(size_t)x * 4 + 3] = table->off_pv[x];
        p->prefix_tokens += (x % H == 0) ? en.n : 0;
        p->logical_bytes += ((int64_t)en.n * (en.rk + en.rv) + (int64_t)(en.rk + en.rv) * d) * 2;
    }
    std::vector<ChunkDev> chunks;
    std::vector<int32_t> g_chunk;
    build_chunks(table, poffs, chunks, g_chunk);
    p->num_chunks = (int)chunks.size();
    for (int g = 0; g < H; ++g)
        p->max_head_chunks = std::max(p->max_head_chunks, g_chunk[(size_t)g + 1] - g_chunk[(size_t)g]);
    // reconstruct-then-attend chunks, in entry order
    std::vector<int4> rc;
    {
        std::vector<int> per_head((size_t)H, 0);
        for (int64_t x = 0; x < E; ++x) {
            const int tiles = (table->block_len[x / H] + kRcTok - 1) / kRcTok;
            for (int t0 = 0; t0 < tiles; t0 += kRcChunkTiles) {
                rc.push_back(make_int4((int)x, t0, std::min(kRcChunkTiles, tiles - t0), 0));
                ++per_head[(size_t)(x % H)];
            }
        }
        p->rc_num_chunks = (int)rc.size();
        for (int g = 0; g < H; ++g) p->rc_max_head_chunks = std::max(p->rc_max_head_chunks, per_head[(size_t)g]);
    }
    // tensor-core path: a partition for every share count sms / ntile that a
    // call with ntile row tiles of kTcRows rows per KV head uses
    p->sms = sms;
    p->tc = !chunks.empty();
    std::vector<TcSegDev> tc_sd;
    std::vector<int32_t> tc_cb;
    if (p->tc) {
        // no share below about one 512-token entry of rank 64 (fewer blocks
        // for small prefixes)
        const TensorCost tcost{table};
        int64_t total = 0;
        for (int64_t x = 0; x < E; ++x) {
            const int n = table->block_len[x / H];
            total += tcost.first((int)x) + tcost.last((int)x);
            for (int t0 = 0; t0 < n; t0 += kTileTokens) total += tcost.tile((int)x, (std::min(n - t0, kTileTokens) + 7) & ~7);
        }
        p->tc_max_shares = (int)std::max<int64_t>(1, std::min<int64_t>(sms, total / kTcMinShareCost));
        const int64_t nt_max = ((int64_t)max_batch * G + kTcRows - 1) / kTcRows;
        std::vector<int> counts;
        for (int64_t nt = 1; nt <= nt_max; ++nt) {
            const int ns = p->tc_shares(nt);
            if (std::find(counts.begin(), counts.end(), ns) == counts.end()) counts.push_back(ns);
            if (ns == 1) break;
        }
        for (int ns : counts) {
            std::vector<Seg> ts;
            std::vector<int32_t> cb;
            int nslot = 0;
            partition_with(table, ns, TensorCost{table}, ts, cb, nslot);
            std::vector<int> runs((size_t)H, 0);
            for (const Seg &x : ts)
                if (x.flags & kSegFirstOfRun) ++runs[(size_t)(x.entry % H)];
            milo_prefix::TcPart tp;
            tp.nshare = ns;
            tp.seg0 = (int)tc_sd.size();
            tp.cta0 = (int)tc_cb.size();
            tp.num_slots = nslot;
            tp.max_runs = *std::max_element(runs.begin(), runs.end());
            for (const Seg &x : ts) {
                const EntryDev &en = ents[(size_t)x.entry];
                tc_sd.push_back(TcSegDev{en.off_ck, en.off_pk, en.off_cv, en.off_pv, x.t0, x.t1, en.n, en.rk, en.rv,
                                         en.g, x.slot, x.flags});
            }
            tc_cb.insert(tc_cb.end(), cb.begin(), cb.end());
            p->tc_parts.push_back(tp);
        }
    }

    int64_t *loff_dev = nullptr;
    auto cleanup = [&](cudaError_t err, const char *what) {
        cudaFree(loff_dev);
        milo_prefix_destroy(p);
        return cuda_fail(err, what);
    };
    // + the accumulators of the chunk grid's calls
    const size_t cnt_bytes = acc_bytes(H, 8 * p->max_nrg, d);
    if ((e = cudaMalloc(&p->packed, (size_t)std::max<int64_t>(p->packed_bytes, 128))) != cudaSuccess)
        return cleanup(e, "cudaMalloc packed");
    if ((e = cudaMalloc(&p->entries, sizeof(EntryDev) * std::max<size_t>(ents.size(), 1))) != cudaSuccess)
        return cleanup(e, "cudaMalloc entries");
    if ((e = cudaMalloc(&p->chunks, sizeof(ChunkDev) * std::max<size_t>(chunks.size(), 1))) != cudaSuccess)
        return cleanup(e, "cudaMalloc chunks");
    if (!chunks.empty() && (e = cudaMemcpyAsync(p->chunks, chunks.data(), sizeof(ChunkDev) * chunks.size(),
                                                cudaMemcpyHostToDevice, stream)) != cudaSuccess)
        return cleanup(e, "copy chunks");
    if (!rc.empty()) {
        if ((e = cudaMalloc(&p->rc_chunks, sizeof(int4) * rc.size())) != cudaSuccess)
            return cleanup(e, "cudaMalloc reconstruction chunks");
        if ((e = cudaMemcpyAsync(p->rc_chunks, rc.data(), sizeof(int4) * rc.size(), cudaMemcpyHostToDevice,
                                 stream)) != cudaSuccess)
            return cleanup(e, "copy reconstruction chunks");
    }
    if ((e = cudaMalloc(&p->acc, cnt_bytes)) != cudaSuccess) return cleanup(e, "cudaMalloc accumulators");
    if ((e = cudaMalloc(&p->status, sizeof(int32_t))) != cudaSuccess) return cleanup(e, "cudaMalloc status");
    if ((e = cudaMalloc(&loff_dev, sizeof(int64_t) * std::max<size_t>(loffs.size(), 1))) != cudaSuccess)
        return cleanup(e, "cudaMalloc offsets");
    if (p->tc) {
        if ((e = cudaMalloc(&p->tc_segs, sizeof(TcSegDev) * tc_sd.size())) != cudaSuccess)
            return cleanup(e, "cudaMalloc tensor-core segments");
        if ((e = cudaMalloc(&p->tc_cta, sizeof(int32_t) * tc_cb.size())) != cudaSuccess)
            return cleanup(e, "cudaMalloc tensor-core shares");
        if ((e = cudaMemcpyAsync(p->tc_segs, tc_sd.data(), sizeof(TcSegDev) * tc_sd.size(), cudaMemcpyHostToDevice,
                                 stream)) != cudaSuccess)
            return cleanup(e, "copy tensor-core segments");
        if ((e = cudaMemcpyAsync(p->tc_cta, tc_cb.data(), sizeof(int32_t) * tc_cb.size(), cudaMemcpyHostToDevice,
                                 stream)) != cudaSuccess)
            return cleanup(e, "copy tensor-core shares");
    }

    if (!ents.empty() &&
        (e = cudaMemcpyAsync(p->entries, ents.data(), sizeof(EntryDev) * ents.size(), cudaMemcpyHostToDevice,
                             stream)) != cudaSuccess)
        return cleanup(e, "copy entries");
    if (!loffs.empty() && (e = cudaMemcpyAsync(loff_dev, loffs.data(), sizeof(int64_t) * loffs.size(),
                                               cudaMemcpyHostToDevice, stream)) != cudaSuccess)
        return cleanup(e, "copy offsets");
    if ((e = cudaMemsetAsync(p->acc, 0, cnt_bytes, stream)) != cudaSuccess) return cleanup(e, "memset accumulators");
    if ((e = cudaMemsetAsync(p->status, 0, sizeof(int32_t), stream)) != cudaSuccess) return cleanup(e, "memset status");
    if ((e = launch_pack(table->arena, p->entries, loff_dev, (int)E, d, p->packed, p->packed_bytes, stream)) !=
        cudaSuccess)
        return cleanup(e, "pack kernel");
    if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cleanup(e, "synchronize after pack");
    cudaFree(loff_dev);
    *out_plan = p;
    return MILO_OK;
}

milo_status_t milo_prefix_get_info(const milo_prefix_t *plan, milo_prefix_info_t *info)
{
    if (!plan || !info) return fail(MILO_ERR_INVALID_ARG, "null argument");
    info->num_blocks = plan->nb;
    info->num_kv_heads = plan->hkv;
    info->num_q_heads = plan->hq;
    info->head_dim = plan->d;
    info->max_batch = plan->max_batch;
    info->prefix_tokens = plan->prefix_tokens;
    info->logical_factor_bytes = plan->logical_bytes;
    info->packed_bytes = plan->packed_bytes;
    info->packed_arena = plan->packed;
    return MILO_OK;
}

namespace {
// An INT8 plan in device memory that is not staged: the chunk grid reads its
// codes directly.
bool reads_int8(const milo_prefix_t *p) { return !p->packed && p->int8_store && !p->int8_host; }

struct CallShape {
    int rows_g, nrg, nrg_t, S;  // query rows and row groups per KV head, row groups per query, tail splits
    int P;         // kTailTokens pieces per tail item
    int path;      // milo_path_t
    int ntile;     // tensor-core path: row tiles per KV head
    const milo_prefix::TcPart *part;
    int64_t records;
    int64_t list_cap, list_bytes;
    // reconstruct-then-attend calls (the same accumulators and finish grid):
    // one record per chunk and row group, then the tail items'
    int64_t records_rc, list_cap_rc, list_bytes_rc;
};

CallShape call_shape(const milo_prefix_t *p, int batch, int64_t max_tail)
{
    CallShape c;
    c.rows_g = batch * p->G;
    c.nrg = (c.rows_g + 7) / 8;
    c.nrg_t = (p->G + 7) / 8;
    // the chunk grid serves every call (a call without a prefix holds tail
    // items alone); its prefix part moves to the tensor cores from
    // kTcMinRows rows per KV head
    c.ntile = 0;
    c.part = nullptr;
    if (p->tc && c.rows_g >= p->tc_min_rows && !reads_int8(p)) {
        c.ntile = (c.rows_g + kTcRows - 1) / kTcRows;
        c.part = p->tc_part(c.ntile);
    }
    c.path = c.part ? MILO_PATH_TENSOR : MILO_PATH_CHUNKS;
    if (!c.part) c.ntile = 0;
    // tail items: on the tensor-core path the chunk grid holds the tails
    // alone, and each item streams up to kTailPiecesLong pieces (fewer items,
    // each merged once); beside prefix chunks an item is one piece
    c.P = c.path == MILO_PATH_TENSOR ? kTailPiecesLong : 1;
    c.S = max_tail > 0 ? (int)((max_tail + (int64_t)c.P * kTailTokens - 1) / ((int64_t)c.P * kTailTokens)) : 0;
    // one record per prefix chunk and row group (the chunk grid), or per run
    // and row group (the tensor-core grid); then the tail items.  Outlier
    // records are listed: int4 [Hkv][nrg][list_cap], list_cap bounding the
    // items whose rows meet one row group: the KV head's chunks (or runs),
    // and the tail items below.
    const int64_t prefix = c.part ? (int64_t)c.part->num_slots * c.nrg : (int64_t)p->num_chunks * c.nrg;
    c.records = prefix + (int64_t)batch * p->hkv * c.S * c.nrg_t;
    // tail items (per split) whose 8 rows meet one row group: with G <= 8 an
    // item is one query's G rows, at most 7 / G + 2 queries meet 8 rows; with
    // G > 8 an item is 8 (or fewer, the query's last) of a query's rows, and
    // at most three such spans meet 8 rows
    const int64_t queries_per_group =
        p->G <= 8 ? std::min<int64_t>(batch, 7 / p->G + 2) : std::min<int64_t>((int64_t)batch * c.nrg_t, 3);
    const int64_t prefix_items = c.part ? (int64_t)c.part->max_runs : (int64_t)p->max_head_chunks;
    c.list_cap = prefix_items + queries_per_group * c.S;
    c.list_bytes = 16 * (int64_t)p->hkv * c.nrg * c.list_cap;
    const int64_t tail_records = (int64_t)batch * p->hkv * c.S * c.nrg_t;
    c.records_rc = (int64_t)p->rc_num_chunks * c.nrg + tail_records;
    c.list_cap_rc = (int64_t)p->rc_max_head_chunks + queries_per_group * c.S;
    c.list_bytes_rc = 16 * (int64_t)p->hkv * c.nrg * c.list_cap_rc;

    return c;
}
}  // namespace

milo_status_t milo_workspace_size(const milo_prefix_t *plan, int32_t batch, int64_t max_tail_tokens, size_t *bytes)
{
    if (!plan || !bytes) return fail(MILO_ERR_INVALID_ARG, "null argument");
    if (batch < 1 || batch > plan->max_batch) return fail(MILO_ERR_INVALID_ARG, "batch outside [1, max_batch]");
    if (max_tail_tokens < 0) return fail(MILO_ERR_INVALID_ARG, "max_tail_tokens < 0");
    const CallShape c = call_shape(plan, batch, max_tail_tokens);
    const size_t rec_bytes = (8 * plan->d + kRecFloatsExtra) * sizeof(float);
    // enough for milo_attn_decode and milo_attn_decode_reconstruct alike
    const size_t a = (size_t)std::max<int64_t>(c.records, 1) * rec_bytes + (size_t)c.list_bytes;
    const size_t b = (size_t)std::max<int64_t>(c.records_rc, 1) * rec_bytes + (size_t)c.list_bytes_rc;
    *bytes = std::max(a, b);
    return MILO_OK;
}

namespace {
// One decode call: the rank-space paths, or (recon) reconstruct-then-attend.
milo_status_t decode_call(const milo_prefix_t *plan, const void *q, int32_t batch, const void *tail_k,
                          const void *tail_v, const int64_t *tail_offsets, int64_t tail_rows, int64_t max_tail_tokens,
                          float softmax_scale, float *out, void *workspace, size_t workspace_bytes, void *stream_,
                          bool recon)
{
    if (!plan || !q || !out) return fail(MILO_ERR_INVALID_ARG, "null plan, q or out");
    if (!recon && plan->rope_tile)
        return fail(MILO_ERR_UNSUPPORTED, "the plan holds pre-RoPE factors: use milo_attn_decode_reconstruct");
    if (!plan->packed && !(reads_int8(plan) && !recon))
        return fail(MILO_ERR_INVALID_ARG, "the plan's arena is offloaded: stage it first (milo_prefix_stage)");
    if (batch < 1 || batch > plan->max_batch) return fail(MILO_ERR_INVALID_ARG, "batch outside [1, max_batch]");
    if (max_tail_tokens < 0) return fail(MILO_ERR_INVALID_ARG, "max_tail_tokens < 0");
    if (plan->nb == 0 && max_tail_tokens == 0) return fail(MILO_ERR_INVALID_ARG, "no prefix and no tail");
    if (max_tail_tokens > 0) {
        if (!tail_k || !tail_v || !tail_offsets) return fail(MILO_ERR_INVALID_ARG, "null tail pointer");
        if (tail_rows < 1 || tail_rows > 0x7fffffff) return fail(MILO_ERR_INVALID_ARG, "tail_rows outside [1, 2^31)");
        if (reinterpret_cast<uintptr_t>(tail_k) % 16 || reinterpret_cast<uintptr_t>(tail_v) % 16)
            return fail(MILO_ERR_ALIGNMENT, "tails must be 16-byte aligned");
        if (max_tail_tokens > (int64_t)kTailTokens * (1 << 20)) return fail(MILO_ERR_INVALID_ARG, "tail too long");
    }
    if (reinterpret_cast<uintptr_t>(q) % 16) return fail(MILO_ERR_ALIGNMENT, "q must be 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(out) % 16) return fail(MILO_ERR_ALIGNMENT, "out must be 16-byte aligned");
    size_t need = 0;
    milo_workspace_size(plan, batch, max_tail_tokens, &need);
    if (!workspace || workspace_bytes < need) return fail(MILO_ERR_WORKSPACE, "workspace missing or too small");
    if (reinterpret_cast<uintptr_t>(workspace) % 16) return fail(MILO_ERR_ALIGNMENT, "workspace misaligned");
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) return fail(MILO_ERR_INVALID_ARG, "plan belongs to another device");

    const CallShape c = call_shape(plan, batch, max_tail_tokens);
    if (recon && plan->rc_num_chunks == 0)
        return fail(MILO_ERR_UNSUPPORTED, "reconstruct-then-attend needs a prefix");
    if (recon && ((int64_t)plan->rc_num_chunks * c.nrg > 0x7fffffff || c.list_cap_rc > 0x7fffffff ||
                  (int64_t)plan->rc_num_chunks * ((c.rows_g + kRcRows - 1) / kRcRows) > 0x7fffffff))
        return fail(MILO_ERR_UNSUPPORTED, "call too large: more than 2^31 - 1 work items");
    // the kernels count thread blocks, tail items and list entries in int
    const int64_t tail_items = (int64_t)batch * plan->hkv * c.S * c.nrg_t;
    if (tail_items > 0x7fffffff || (int64_t)plan->num_chunks * c.nrg + tail_items > 0x7fffffff ||
        c.list_cap > 0x7fffffff || (int64_t)plan->hkv * c.nrg > 0x7fffffff)
        return fail(MILO_ERR_UNSUPPORTED, "call too large: more than 2^31 - 1 work items");
    DecodeParams prm{};
    prm.packed = plan->packed;
    if (reads_int8(plan)) {
        prm.q8_codes = plan->int8_dev;
        prm.q8_params = reinterpret_cast<const uint32_t *>(plan->int8_dev + plan->packed_bytes / 2);
    }
    prm.entries = plan->entries;
    prm.q = static_cast<const uint16_t *>(q);
    prm.tail_offsets = tail_offsets;
    prm.out = out;
    prm.rec = static_cast<float *>(workspace);

    {
        // reference maxima, list counts, then the 16-byte aligned sums and
        // output accumulators
        const int H = plan->hkv, R = 8 * plan->max_nrg;
        prm.rows_max = R;
        prm.acc_m = reinterpret_cast<uint32_t *>(plan->acc);
        prm.ovf_cnt = prm.acc_m + (size_t)H * R;
        prm.acc_l = reinterpret_cast<float *>(plan->acc + acc_l_offset(H, R));
        prm.acc_o = prm.acc_l + (size_t)H * R;
    }
    prm.status = plan->status;
    prm.batch = batch;
    prm.hq = plan->hq;
    prm.hkv = plan->hkv;
    prm.G = plan->G;
    prm.d = plan->d;
    prm.rows_g = c.rows_g;
    prm.nrg = c.nrg;
    prm.nrg_t = c.nrg_t;
    prm.tail_splits = c.S;
    prm.tail_pieces = c.P;
    prm.num_tail_items = (int)tail_items;
    prm.has_tail = c.S > 0 ? 1 : 0;
    prm.tail_k = static_cast<const uint16_t *>(tail_k);
    prm.tail_v = static_cast<const uint16_t *>(tail_v);
    prm.chunks = plan->chunks;
    prm.num_chunks = c.path == MILO_PATH_CHUNKS ? plan->num_chunks : 0;
    if (c.part) {
        prm.tc_segs = plan->tc_segs + c.part->seg0;
        prm.tc_cta_begin = plan->tc_cta + c.part->cta0;
        prm.tc_ntile = c.ntile;
        prm.tc_nshare = c.part->nshare;
    }
    {
        prm.tail_rec_base = c.part ? (int64_t)c.part->num_slots * c.nrg : (int64_t)plan->num_chunks * c.nrg;
        // the record lists follow the records
        prm.list_cap = (int)c.list_cap;
        prm.ovf_list = reinterpret_cast<int32_t *>(static_cast<uint8_t *>(workspace) +
                                                   (size_t)c.records * (8 * plan->d + kRecFloatsExtra) * sizeof(float));
    }
    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt((float)plan->d);
    prm.scale_log2 = scale * 1.4426950408889634f;

    alignas(64) CUtensorMap mk, mv;
    std::memset(&mk, 0, sizeof mk);
    std::memset(&mv, 0, sizeof mv);
    if (c.S > 0) {
        EncodeTiledFn enc = encode_fn();
        if (!enc) return fail(MILO_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
        const cuuint64_t dims[3] = {(cuuint64_t)plan->d, (cuuint64_t)plan->hkv, (cuuint64_t)tail_rows};
        const cuuint64_t strides[2] = {(cuuint64_t)plan->d * 2, (cuuint64_t)plan->hkv * plan->d * 2};
        // the chunk grid's tail items: boxes of 64 columns (128-byte rows,
        // 128-byte swizzle), few wide requests
        const cuuint32_t box[3] = {64u, 1, (cuuint32_t)kTailTokens};
        const cuuint32_t estr[3] = {1, 1, 1};
        const CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B;
        CUresult r1 = enc(&mk, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(tail_k), dims, strides, box,
                          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        CUresult r2 = enc(&mv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(tail_v), dims, strides, box,
                          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r1 != CUDA_SUCCESS || r2 != CUDA_SUCCESS) return fail(MILO_ERR_CUDA, "tensor map encoding failed");
    }
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    if (recon) {
        // the dense tails on the chunk grid, then the reconstructing prefix
        // grid, then the finish grid (each chained by programmatic dependent
        // launch); records: the chunks' first, then the tail items'
        prm.num_chunks = 0;
        prm.tc_ntile = 0;
        prm.rc_chunks = plan->rc_chunks;
        prm.rope_tile = plan->rope_tile;
        prm.rope_off = plan->rope_off;
        prm.rope_tile_base = plan->rope_tile_base;
        prm.tail_rec_base = (int64_t)plan->rc_num_chunks * c.nrg;
        prm.list_cap = (int)c.list_cap_rc;
        prm.ovf_list = reinterpret_cast<int32_t *>(static_cast<uint8_t *>(workspace) +
                                                   (size_t)std::max<int64_t>(c.records_rc, 1) *
                                                       (8 * plan->d + kRecFloatsExtra) * sizeof(float));
        cudaError_t e = cudaSuccess;
        if (prm.num_tail_items > 0 && (e = launch_chunks(prm, &mk, &mv, stream)) != cudaSuccess)
            return cuda_fail(e, "tail grid launch");
        if ((e = launch_recon(prm, plan->rc_num_chunks, stream)) != cudaSuccess)
            return cuda_fail(e, "reconstruction grid launch");
        if ((e = launch_finish(prm, stream)) != cudaSuccess) return cuda_fail(e, "finish grid launch");
        return MILO_OK;
    }
    if (c.path == MILO_PATH_TENSOR) {
        // the dense tails on the chunk grid, then the prefix on the tensor
        // cores, then the finish grid (each chained by programmatic
        // dependent launch)
        cudaError_t e = cudaSuccess;
        if (prm.num_tail_items > 0 && (e = launch_chunks(prm, &mk, &mv, stream)) != cudaSuccess)
            return cuda_fail(e, "tail grid launch");
        if ((e = launch_batch_tc(prm, stream)) != cudaSuccess) return cuda_fail(e, "tensor-core grid launch");
        if ((e = launch_finish(prm, stream)) != cudaSuccess) return cuda_fail(e, "finish grid launch");
        return MILO_OK;
    }
    // MILO_PATH_CHUNKS: the prefix chunks and the tail items in one grid
    // (tail items alone without a prefix), then the finish grid
    cudaError_t e = launch_chunks(prm, &mk, &mv, stream);
    if (e != cudaSuccess) return cuda_fail(e, "chunk grid launch");
    return MILO_OK;
}
}  // namespace

milo_status_t milo_attn_decode(const milo_prefix_t *plan, const void *q, int32_t batch, const void *tail_k,
                               const void *tail_v, const int64_t *tail_offsets, int64_t tail_rows,
                               int64_t max_tail_tokens, float softmax_scale, float *out, void *workspace,
                               size_t workspace_bytes, void *stream)
{
    return decode_call(plan, q, batch, tail_k, tail_v, tail_offsets, tail_rows, max_tail_tokens, softmax_scale, out,
                       workspace, workspace_bytes, stream, false);
}

milo_status_t milo_attn_decode_reconstruct(const milo_prefix_t *plan, const void *q, int32_t batch,
                                           const void *tail_k, const void *tail_v, const int64_t *tail_offsets,
                                           int64_t tail_rows, int64_t max_tail_tokens, float softmax_scale,
                                           float *out, void *workspace, size_t workspace_bytes, void *stream)
{
    return decode_call(plan, q, batch, tail_k, tail_v, tail_offsets, tail_rows, max_tail_tokens, softmax_scale, out,
                       workspace, workspace_bytes, stream, true);
}

milo_status_t milo_prefix_set_rope(milo_prefix_t *plan, double rope_theta, const int64_t *block_pos)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    if (!(rope_theta >= 0.0) || std::isinf(rope_theta)) return fail(MILO_ERR_INVALID_ARG, "rope_theta must be finite and >= 0");
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) return fail(MILO_ERR_INVALID_ARG, "plan belongs to another device");
    cudaError_t e = cudaDeviceSynchronize();  // no call may be reading the old tables
    if (e != cudaSuccess) return cuda_fail(e, "synchronize before the rotation tables change");
    cudaFree(plan->rope_tile);
    cudaFree(plan->rope_off);
    cudaFree(plan->rope_tile_base);
    plan->rope_tile = plan->rope_off = nullptr;
    plan->rope_tile_base = nullptr;
    if (rope_theta == 0.0) return MILO_OK;
    const int d = plan->d, h = d / 2, nb = plan->nb;
    if (!plan->rc_chunks) return fail(MILO_ERR_UNSUPPORTED, "no prefix to rotate");
    // block positions (default: the blocks' starts in the concatenated prefix)
    std::vector<int32_t> len((size_t)nb);
    std::vector<int32_t> base((size_t)nb + 1, 0);
    {
        std::vector<EntryDev> ents((size_t)nb * plan->hkv);
        if ((e = cudaMemcpy(ents.data(), plan->entries, sizeof(EntryDev) * ents.size(), cudaMemcpyDeviceToHost)) !=
            cudaSuccess)
            return cuda_fail(e, "read the plan's entries");
        for (int b = 0; b < nb; ++b) len[(size_t)b] = ents[(size_t)b * plan->hkv].n;
    }
    std::vector<int64_t> pos((size_t)nb);
    int64_t cum = 0;
    for (int b = 0; b < nb; ++b) {
        pos[(size_t)b] = block_pos ? block_pos[b] : cum;
        if (pos[(size_t)b] < 0 || pos[(size_t)b] > ((int64_t)1 << 40))
            return fail(MILO_ERR_INVALID_ARG, "block position outside [0, 2^40]");
        cum += len[(size_t)b];
        base[(size_t)b + 1] = base[(size_t)b] + (len[(size_t)b] + kRcTok - 1) / kRcTok;
    }
    // frequency of pair i, and the (cos, sin) tables, in fp64 then rounded
    std::vector<double> th((size_t)h);
    for (int i = 0; i < h; ++i) th[(size_t)i] = std::pow(rope_theta, -2.0 * i / d);
    std::vector<float2> off((size_t)kRcTok * h), tile((size_t)base[(size_t)nb] * h);
    for (int u = 0; u < kRcTok; ++u)
        for (int i = 0; i < h; ++i) {
            const double a = u * th[(size_t)i];
            off[(size_t)u * h + i] = make_float2((float)std::cos(a), (float)std::sin(a));
        }
    for (int b = 0; b < nb; ++b)
        for (int k = 0; k < base[(size_t)b + 1] - base[(size_t)b]; ++k)
            for (int i = 0; i < h; ++i) {
                const double a = (double)(pos[(size_t)b] + (int64_t)k * kRcTok) * th[(size_t)i];
                tile[((size_t)base[(size_t)b] + k) * h + i] = make_float2((float)std::cos(a), (float)std::sin(a));
            }
    auto undo = [&](cudaError_t err, const char *what) {
        cudaFree(plan->rope_tile);
        cudaFree(plan->rope_off);
        cudaFree(plan->rope_tile_base);
        plan->rope_tile = plan->rope_off = nullptr;
        plan->rope_tile_base = nullptr;
        return cuda_fail(err, what);
    };
    if ((e = cudaMalloc(&plan->rope_tile, sizeof(float2) * std::max<size_t>(tile.size(), 1))) != cudaSuccess)
        return undo(e, "cudaMalloc rotation table");
    if ((e = cudaMalloc(&plan->rope_off, sizeof(float2) * off.size())) != cudaSuccess)
        return undo(e, "cudaMalloc rotation table");
    if ((e = cudaMalloc(&plan->rope_tile_base, sizeof(int32_t) * base.size())) != cudaSuccess)
        return undo(e, "cudaMalloc rotation table");
    if ((e = cudaMemcpy(plan->rope_tile, tile.data(), sizeof(float2) * tile.size(), cudaMemcpyHostToDevice)) !=
            cudaSuccess ||
        (e = cudaMemcpy(plan->rope_off, off.data(), sizeof(float2) * off.size(), cudaMemcpyHostToDevice)) !=
            cudaSuccess ||
        (e = cudaMemcpy(plan->rope_tile_base, base.data(), sizeof(int32_t) * base.size(), cudaMemcpyHostToDevice)) !=
            cudaSuccess)
        return undo(e, "copy rotation tables");
    return MILO_OK;
}

milo_status_t milo_call_info(const milo_prefix_t *plan, int32_t batch, int64_t max_tail_tokens,
                             milo_call_info_t *info)
{
    if (!plan || !info) return fail(MILO_ERR_INVALID_ARG, "null argument");
    if (batch < 1 || batch > plan->max_batch) return fail(MILO_ERR_INVALID_ARG, "batch outside [1, max_batch]");
    if (max_tail_tokens < 0) return fail(MILO_ERR_INVALID_ARG, "max_tail_tokens < 0");
    const CallShape c = call_shape(plan, batch, max_tail_tokens);
    info->path = c.path;
    info->row_tiles = c.ntile;
    if (c.path == MILO_PATH_TENSOR) {
        info->kernels = (c.S > 0 ? 1 : 0) + 2;
        info->blocks = c.part->nshare * c.ntile;
    } else {
        info->kernels = 2;
        const int rg = c.nrg >= 2 ? 2 : 1;
        const int64_t tail_items = (int64_t)batch * plan->hkv * c.S * c.nrg_t;
        info->blocks = (int32_t)std::min<int64_t>(
            (int64_t)plan->num_chunks * ((c.nrg + rg - 1) / rg) + (tail_items + rg - 1) / rg, 0x7fffffff);
    }
    return MILO_OK;
}

int32_t milo_tensor_min_rows(void) { return kTcMinRows; }

milo_status_t milo_prefix_set_tensor_min_rows(milo_prefix_t *plan, int32_t rows)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    if (rows < 1) return fail(MILO_ERR_INVALID_ARG, "rows < 1");
    plan->tc_min_rows = rows;
    return MILO_OK;
}

milo_status_t milo_attn_decode_static(const milo_prefix_t *plan, const void *q, int32_t batch,
                                      const void *tail_k, const void *tail_v, const int64_t *tail_offsets,
                                      int64_t tail_rows, int64_t max_tail_tokens, float softmax_scale, float *out,
                                      void *stream)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    size_t need = 0;
    milo_status_t s = milo_workspace_size(plan, batch, max_tail_tokens, &need);
    if (s != MILO_OK) return s;
    if (need > kStaticWorkspaceBytes)
        return fail(MILO_ERR_WORKSPACE, "call needs " + std::to_string(need) +
                                            " bytes of scratch; the built-in scratch holds " +
                                            std::to_string(kStaticWorkspaceBytes) + " (use milo_attn_decode)");
    void *ws = nullptr;
    cudaError_t e = static_workspace(&ws);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the built-in scratch");
    return milo_attn_decode(plan, q, batch, tail_k, tail_v, tail_offsets, tail_rows, max_tail_tokens,
                            softmax_scale, out, ws, kStaticWorkspaceBytes, stream);
}

namespace {
// Checks of an encode request; on success the starting ranks fit both budgets.
milo_status_t check_encode(const milo_encode_params_t *q)
{
    if (!q || !q->block_len) return fail(MILO_ERR_INVALID_ARG, "null encode parameters");
    if (q->num_blocks < 1 || q->num_kv_heads < 1) return fail(MILO_ERR_INVALID_ARG, "no blocks or no KV heads");
    if (q->head_dim != 64 && q->head_dim != 128) return fail(MILO_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (q->r_min < 0 || q->r_max < q->r_min) return fail(MILO_ERR_INVALID_ARG, "need 0 <= r_min <= r_max");
    if ((int64_t)q->num_blocks * q->num_kv_heads * 2 > 0x7fffffff) return fail(MILO_ERR_UNSUPPORTED, "too many blocks");
    int64_t start = 0;
    for (int b = 0; b < q->num_blocks; ++b) {
        const int n = q->block_len[b];
        if (n < 1 || n > 65536) return fail(MILO_ERR_BAD_TABLE, "block length outside [1, 65536]");
        start += std::min(q->r_min, std::min(n, q->head_dim));
    }
    if (q->budget_k < start || q->budget_v < start)
        return fail(MILO_ERR_INVALID_ARG, "a budget is below the starting ranks sum(min(r_min, n_b, d))");
    return MILO_OK;
}
// Workspace of an encode: block starts and lengths, the layout, the status
// word, the singular values and the eigenvectors.
struct EncodeWs {
    size_t tok0, blen, offs, status, sigma, vt, total;
};
EncodeWs encode_ws(const milo_encode_params_t *q)
{
    const int64_t nb = q->num_blocks, E = nb * q->num_kv_heads, d = q->head_dim;
    EncodeWs w;
    size_t cur = 0;
    auto take = [&](size_t bytes) {
        const size_t at = cur;
        cur = (cur + bytes + 255) / 256 * 256;
        return at;
    };
    w.tok0 = take(8 * nb);
    w.blen = take(4 * nb);
    w.offs = take(8 * 4 * E);
    w.status = take(16);
    w.sigma = take(4 * 2 * E * d);
    w.vt = take(4 * 2 * E * d * d);
    w.total = cur;
    return w;
}
}  // namespace

milo_status_t milo_encode_layout(const milo_encode_params_t *params, int64_t *offsets, int64_t *arena_elems)
{
    milo_status_t s = check_encode(params);
    if (s != MILO_OK) return s;
    const int64_t n = encode_layout(params->num_blocks, params->num_kv_heads, params->head_dim, params->block_len,
                                    params->r_max, offsets);
    if (arena_elems) *arena_elems = n;
    return MILO_OK;
}

milo_status_t milo_encode_workspace_size(const milo_encode_params_t *params, size_t *bytes)
{
    if (!bytes) return fail(MILO_ERR_INVALID_ARG, "null argument");
    milo_status_t s = check_encode(params);
    if (s != MILO_OK) return s;
    *bytes = encode_ws(params).total;
    return MILO_OK;
}

milo_status_t milo_encode(const milo_encode_params_t *params, const void *k, const void *v, void *arena,
                          int64_t arena_elems, int32_t *rank_k, int32_t *rank_v, float *sigma, void *workspace,
                          size_t workspace_bytes, void *stream_)
{
    milo_status_t s = check_encode(params);
    if (s != MILO_OK) return s;
    if (!k || !v || !arena || !rank_k || !rank_v || !workspace) return fail(MILO_ERR_INVALID_ARG, "null pointer");
    if (reinterpret_cast<uintptr_t>(k) % 16 || reinterpret_cast<uintptr_t>(v) % 16 ||
        reinterpret_cast<uintptr_t>(arena) % 16 || reinterpret_cast<uintptr_t>(workspace) % 256)
        return fail(MILO_ERR_ALIGNMENT, "k, v and arena must be 16-byte aligned, the workspace 256-byte aligned");
    const EncodeWs w = encode_ws(params);
    if (workspace_bytes < w.total) return fail(MILO_ERR_WORKSPACE, "workspace too small");
    const int nb = params->num_blocks, H = params->num_kv_heads, d = params->head_dim;
    std::vector<int64_t> tok0((size_t)nb), offs((size_t)nb * H * 4);
    int64_t cum = 0;
    for (int b = 0; b < nb; ++b) {
        tok0[(size_t)b] = cum;
        cum += params->block_len[b];
    }
    if (cum * H * d > ((int64_t)1 << 40)) return fail(MILO_ERR_UNSUPPORTED, "prefix too long");
    const int64_t need = encode_layout(nb, H, d, params->block_len, params->r_max, offs.data());
    if (arena_elems < need) return fail(MILO_ERR_INVALID_ARG, "arena smaller than milo_encode_layout's count");
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t stream = static_cast<cudaStream_t>(stream_);
    cudaError_t e;
    if ((e = cudaMemcpyAsync(ws + w.tok0, tok0.data(), 8 * tok0.size(), cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(ws + w.blen, params->block_len, 4 * (size_t)nb, cudaMemcpyHostToDevice, stream)) !=
            cudaSuccess ||
        (e = cudaMemcpyAsync(ws + w.offs, offs.data(), 8 * offs.size(), cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaMemsetAsync(ws + w.status, 0, 16, stream)) != cudaSuccess)
        return cuda_fail(e, "stage encode tables");
    // (the copies read host memory that lives until this function returns:
    // wait for them)
    if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cuda_fail(e, "synchronize encode tables");
    float *sg = sigma ? sigma : reinterpret_cast<float *>(ws + w.sigma);
    e = launch_encode(static_cast<const uint16_t *>(k), static_cast<const uint16_t *>(v),
                      reinterpret_cast<const int64_t *>(ws + w.tok0), reinterpret_cast<const int32_t *>(ws + w.blen),
                      reinterpret_cast<const int64_t *>(ws + w.offs), static_cast<uint16_t *>(arena), rank_k, rank_v, sg,
                      reinterpret_cast<float *>(ws + w.vt), reinterpret_cast<int32_t *>(ws + w.status), nb, H, d,
                      params->r_min, params->r_max, params->budget_k, params->budget_v, stream);
    if (e != cudaSuccess) return cuda_fail(e, "encode launch");
    return MILO_OK;
}

milo_status_t milo_prefix_offload(milo_prefix_t *plan)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    if (plan->packed_host) return fail(MILO_ERR_INVALID_ARG, "the plan is already offloaded");
    if (plan->int8_store) return fail(MILO_ERR_INVALID_ARG, "the plan's arena is held as INT8");
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) return fail(MILO_ERR_INVALID_ARG, "plan belongs to another device");
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "synchronize before offloading");
    const size_t bytes = (size_t)std::max<int64_t>(plan->packed_bytes, 128);
    uint8_t *host = nullptr;
    if ((e = cudaHostAlloc(reinterpret_cast<void **>(&host), bytes, cudaHostAllocDefault)) != cudaSuccess)
        return cuda_fail(e, "cudaHostAlloc for the offloaded arena");
    if ((e = cudaMemcpy(host, plan->packed, bytes, cudaMemcpyDeviceToHost)) != cudaSuccess) {
        cudaFreeHost(host);
        return cuda_fail(e, "copy the arena to host memory");
    }
    cudaFree(plan->packed);
    plan->packed = nullptr;
    plan->packed_host = host;
    return MILO_OK;
}

milo_status_t milo_prefix_stage(milo_prefix_t *plan, void *device_buffer, size_t bytes, void *stream)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    if (!device_buffer) {
        // an INT8 plan in device memory goes back to reading its codes
        if (!plan->int8_store || plan->int8_host)
            return fail(MILO_ERR_INVALID_ARG, "null buffer (only an INT8 plan in device memory reads without one)");
        plan->packed = nullptr;
        return MILO_OK;
    }
    if (!plan->packed_host && !plan->int8_store) return fail(MILO_ERR_INVALID_ARG, "the plan is not offloaded");
    if ((int64_t)bytes < plan->packed_bytes) return fail(MILO_ERR_INVALID_ARG, "staging buffer smaller than the arena");
    if (reinterpret_cast<uintptr_t>(device_buffer) % 128) return fail(MILO_ERR_ALIGNMENT, "staging buffer not 128-byte aligned");
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) return fail(MILO_ERR_INVALID_ARG, "plan belongs to another device");
    cudaError_t e;
    if (plan->int8_store) {
        const uint8_t *codes = plan->int8_dev;
        e = launch_dequant_plan_int8(plan->entries, plan->nb * plan->hkv, plan->d, plan->max_factor_groups, codes,
                                     codes + plan->packed_bytes / 2,
                                     device_buffer, static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess) return cuda_fail(e, "stage the INT8 arena");
    } else {
        e = cudaMemcpyAsync(device_buffer, plan->packed_host, (size_t)plan->packed_bytes, cudaMemcpyHostToDevice,
                            static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess) return cuda_fail(e, "stage the arena");
    }
    plan->packed = static_cast<uint8_t *>(device_buffer);
    return MILO_OK;
}

namespace {
milo_status_t check_int8_args(const void *a, const void *b, const void *c, int64_t bytes)
{
    if (!a || !b || !c) return fail(MILO_ERR_INVALID_ARG, "null pointer");
    if (bytes < 0 || bytes % 128) return fail(MILO_ERR_INVALID_ARG, "bytes negative or not a multiple of 128");
    return MILO_OK;
}
}  // namespace

milo_status_t milo_quantize_int8(const void *packed, int64_t bytes, void *codes, void *params, void *stream)
{
    milo_status_t s = check_int8_args(packed, codes, params, bytes);
    if (s != MILO_OK) return s;
    if (reinterpret_cast<uintptr_t>(packed) % 16 || reinterpret_cast<uintptr_t>(codes) % 8 ||
        reinterpret_cast<uintptr_t>(params) % 4)
        return fail(MILO_ERR_ALIGNMENT, "packed not 16-byte, codes not 8-byte or params not 4-byte aligned");
    cudaError_t e = launch_quant_int8(packed, bytes / 128, codes, params, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? MILO_OK : cuda_fail(e, "quantise launch");
}

milo_status_t milo_dequantize_int8(const void *codes, const void *params, int64_t bytes, void *packed, void *stream)
{
    milo_status_t s = check_int8_args(codes, params, packed, bytes);
    if (s != MILO_OK) return s;
    if (reinterpret_cast<uintptr_t>(packed) % 16 || reinterpret_cast<uintptr_t>(codes) % 8 ||
        reinterpret_cast<uintptr_t>(params) % 4)
        return fail(MILO_ERR_ALIGNMENT, "packed not 16-byte, codes not 8-byte or params not 4-byte aligned");
    cudaError_t e = launch_dequant_int8(codes, params, bytes / 128, packed, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? MILO_OK : cuda_fail(e, "dequantise launch");
}

milo_status_t milo_prefix_quantize_int8(milo_prefix_t *plan, int32_t to_host)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    if (plan->packed_host) return fail(MILO_ERR_INVALID_ARG, "the plan is offloaded");
    if (plan->int8_store) return fail(MILO_ERR_INVALID_ARG, "the plan is already held as INT8");
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) return fail(MILO_ERR_INVALID_ARG, "plan belongs to another device");
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "synchronize before quantising");
    const int64_t nbytes = plan->packed_bytes;
    // (+16: the chunk grid copies parameter words in aligned groups of four,
    // which may reach up to three words past the last)
    const size_t store = (size_t)std::max<int64_t>(nbytes / 2 + nbytes / 32, 128) + 16;
    uint8_t *mem = nullptr;
    void *dev = nullptr;
    if (to_host) {
        if ((e = cudaHostAlloc(reinterpret_cast<void **>(&mem), store, cudaHostAllocMapped)) != cudaSuccess)
            return cuda_fail(e, "cudaHostAlloc for the INT8 arena");
        if ((e = cudaHostGetDevicePointer(&dev, mem, 0)) != cudaSuccess) {
            cudaFreeHost(mem);
            return cuda_fail(e, "device address of the INT8 arena");
        }
    } else {
        if ((e = cudaMalloc(reinterpret_cast<void **>(&mem), store)) != cudaSuccess)
            return cuda_fail(e, "cudaMalloc for the INT8 arena");
        dev = mem;
    }
    uint8_t *codes = static_cast<uint8_t *>(dev);
    e = launch_quant_int8(plan->packed, nbytes / 128, codes, codes + nbytes / 2, nullptr);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        if (to_host) cudaFreeHost(mem);
        else cudaFree(mem);
        return cuda_fail(e, "quantise the arena");
    }
    cudaFree(plan->packed);
    plan->packed = nullptr;
    plan->int8_store = mem;
    plan->int8_dev = codes;
    plan->int8_host = to_host != 0;
    return MILO_OK;
}

milo_status_t milo_prefix_storage_bytes(const milo_prefix_t *plan, int64_t *bytes, int32_t *int8, int32_t *on_host)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    const int64_t nb = plan->packed_bytes;
    if (bytes) *bytes = plan->int8_store ? nb / 2 + nb / 32 : nb;
    if (int8) *int8 = plan->int8_store ? 1 : 0;
    if (on_host) *on_host = (plan->packed_host || (plan->int8_store && plan->int8_host)) ? 1 : 0;
    return MILO_OK;
}

milo_status_t milo_check_bounded_wait(const milo_prefix_t *plan, int64_t limit_ns, int32_t arrive, void *stream)
{
    if (!plan) return fail(MILO_ERR_INVALID_ARG, "null plan");
    if (limit_ns < 1000000 || limit_ns > 10000000000LL) return fail(MILO_ERR_INVALID_ARG, "limit_ns outside [1e6, 1e10]");
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != plan->device) return fail(MILO_ERR_INVALID_ARG, "plan belongs to another device");
    cudaError_t e = launch_wait_check(plan->status, (uint64_t)limit_ns, arrive ? 1 : 0, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "wait check launch");
    return MILO_OK;
}

milo_status_t milo_get_device_status(const milo_prefix_t *plan, void *stream, int32_t clear, int32_t *code)
{
    if (!plan || !code) return fail(MILO_ERR_INVALID_ARG, "null argument");
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int32_t v = 0;
    if ((e = cudaMemcpy(&v, plan->status, sizeof v, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_fail(e, "read status");
    *code = v;
    if (clear && (e = cudaMemset(plan->status, 0, sizeof(int32_t))) != cudaSuccess)
        return cuda_fail(e, "clear status");
    return MILO_OK;
}

}  // extern "C"
