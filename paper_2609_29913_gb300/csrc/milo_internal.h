// milo_internal.h -- structures shared by the libmilo host code and kernels.
#pragma once
#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace milo {

constexpr int kTileTokens = 32;      // tokens per partition cut (the tensor-core grid's segments)
constexpr int kTailTokens = 64;      // tokens per dense-tail work item (per piece of one)
constexpr int kTailPiecesLong = 8;   // pieces per tail item when the chunk grid holds tails alone
constexpr int kRecFloatsExtra = 16;  // m[8], l[8] after o[8][d] in a record

// Per-(block, KV head) entry of the packed arena.
struct EntryDev {
    int64_t off_ck, off_pk, off_cv, off_pv;  // byte offsets (128-aligned)
    int32_t n;                               // tokens
    int32_t rk, rv;                          // true ranks
    int32_t g;                               // KV head
};

// Flags of a segment of the tensor-core grid's partition.
enum : int32_t { kSegFirstOfRun = 1, kSegLastOfRun = 2 };

// One chunk of the chunk grid: tokens [t0, t1) of a prefix entry.
constexpr int kChunkBytes = 131072;   // coefficient bytes (C^K + C^V rows) per chunk
constexpr int kChunkMaxTok = 1024;   // tokens per chunk
struct ChunkDev {
    int64_t ck, cv, pk, pv;     // byte offsets in the packed arena (C^K, C^V at the chunk's first token)
    int32_t ntok, tok8;         // tokens, and rows copied (rounded up to 8 within the entry)
    int32_t nrk, nrv;           // rank 8-groups of K and V
    int32_t g;                  // KV head
    int32_t rk, rv;             // true ranks (the INT8 read zeroes P rows past them)
    int32_t pad;
};
static_assert(sizeof(ChunkDev) == 64, "chunk descriptor size");

// The tensor-core prefix decode (milo_batch.cu): query rows per tile (the M
// side of its products), tokens per score tile, bytes per ring slot, and the
// query rows per KV head from which a call takes it.
constexpr int kTcRows = 128;
constexpr int kTcTok = 64;
constexpr int kTcSlot = 32768;
constexpr int kTcMinRows = 32;

// A segment of the tensor-core decode's partition, with what it needs of its
// entry (one 64-byte load, no dependent loads).
struct TcSegDev {
    int64_t ck, pk, cv, pv;     // packed byte offsets of the entry's factors
    int32_t t0, t1;             // tokens [t0, t1) of the entry
    int32_t n, rk, rv, g;       // entry tokens, ranks, KV head
    int32_t slot, flags;        // run record slot, kSegFirstOfRun / kSegLastOfRun
};
static_assert(sizeof(TcSegDev) == 64, "tensor-core segment size");

// Reconstruct-then-attend (milo_recon.cu): tokens per reconstructed tile,
// query rows per thread block, and tiles per chunk (a chunk is a thread
// block's token range of one entry: int4 {entry, first tile, tiles, 0}).
constexpr int kRcTok = 64;
constexpr int kRcRows = 128;
constexpr int kRcChunkTiles = 4;

struct DecodeParams {
    const uint8_t *packed;
    const EntryDev *entries;
    const uint16_t *q;              // bf16 [batch, Hq, d]
    const int64_t *tail_offsets;    // [batch + 1] or null
    float *out;                     // [batch, Hq, d]
    float *rec;                     // workspace records
    int32_t *status;
    int batch, hq, hkv, G, d;
    int rows_g;                     // batch * G
    int nrg;                        // ceil(rows_g / 8)
    int nrg_t;                      // tail row groups per query: ceil(G / 8)
    int tail_splits;                // S: tail items per (query, KV head)
    int tail_pieces;                // kTailTokens pieces per tail item (the chunk grid)
    int num_tail_items;             // batch * Hkv * S * nrg_t
    int has_tail;
    int64_t tail_rec_base;          // first tail record index
    float scale_log2;               // softmax scale * log2(e)
    const ChunkDev *chunks;         // the chunk grid's prefix chunks (KV-head-major)
    const uint8_t *q8_codes;        // INT8 plan read directly (packed is then null): core i's 64 codes
    const uint32_t *q8_params;      //   at q8_codes + 64 i, its parameter word at q8_params[i]
    int num_chunks;                 // prefix chunks in this call's chunk grid (0: tail items alone)
    const uint16_t *tail_k, *tail_v;  // bf16 [rows, Hkv, d] dense tails (or null)
    int rows_max;                   // accumulator rows per KV head: 8 ceil(max_batch G / 8)
    float *acc_o;                   // [Hkv][rows_max][d]: per-row accumulators of the call
    float *acc_l;                   // [Hkv][rows_max]
    uint32_t *acc_m;                // [Hkv][rows_max]: reference maxima (sign-flipped float bits; 0 = unset)
    uint32_t *ovf_cnt;              // [Hkv][nrg]: records listed per (KV head, row group)
    int32_t *ovf_list;              // int4 [Hkv][nrg][list_cap]: listed records (workspace)
    int list_cap;                   // list entries per (KV head, row group)
    const TcSegDev *tc_segs;        // tensor-core path: segments of this call's partition
    const int32_t *tc_cta_begin;    //   [tc_nshare + 1] first segment of each share
    int tc_ntile;                   //   tiles of kTcRows query rows per KV head
    int tc_nshare;                  //   shares (thread blocks per row tile)
    const int4 *rc_chunks;          // reconstruct-then-attend: the prefix chunks (or null)
    const float2 *rope_tile;        //   pre-RoPE factors: (cos, sin) of each tile start's angle, [tile][d/2]
    const float2 *rope_off;         //   (cos, sin) of u theta_i for u < kRcTok, [u][d/2]
    const int32_t *rope_tile_base;  //   first tile of each block in rope_tile
};

// Kernel attributes (shared-memory size, carveout) belong to a device: the
// launchers set them once per device, tracked in tables of kMaxDevices.
constexpr int kMaxDevices = 64;
// The current device, or -1 when it cannot be read or lies past the tables
// (the caller then sets the attributes on every launch).
inline int attribute_slot()
{
    int d = -1;
    if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
    return d;
}

// Launchers implemented in the .cu files.
cudaError_t launch_pack(const void *arena, const EntryDev *entries_dev,
                        const int64_t *logical_offsets_dev, int num_entries,
                        int head_dim, uint8_t *packed, int64_t packed_bytes,
                        cudaStream_t stream);

// The chunk grid (one thread block per prefix chunk and row group of 8 query
// rows, and per tail item), then its finish grid.
cudaError_t launch_chunks(const DecodeParams &p, const void *tmap_k, const void *tmap_v, cudaStream_t stream);


// The tensor-core prefix grid (a thread block per share and row tile); the
// call's tail items run on the chunk grid before it, and its finish grid
// after it.
cudaError_t launch_batch_tc(const DecodeParams &p, cudaStream_t stream);
int batch_tc_smem_bytes(int head_dim);
// The finish grid alone (one warp per KV head and row group).
cudaError_t launch_finish(const DecodeParams &p, cudaStream_t stream);
// The reconstruct-then-attend prefix grid (a thread block per chunk and group
// of kRcRows query rows); like the tensor-core grid it sits between the tail
// items' chunk grid and the finish grid.
cudaError_t launch_recon(const DecodeParams &p, int num_chunks, cudaStream_t stream);
// One warp's bounded wait on an mbarrier that nothing completes (arrive = 0)
// or that it completes first (arrive = 1), against a status word.
cudaError_t launch_wait_check(int32_t *status, uint64_t limit_ns, int arrive, cudaStream_t stream);

// The compression stage (milo_encode.cu): the arena layout of its output
// (element offsets [E][4] of C^K, P^K, C^V, P^V, each region sized for
// min(r_max, n_b, d) ranks and 8-element aligned; returns the element
// count), and the launch of its three grids.
int64_t encode_layout(int nb, int hkv, int d, const int32_t *blen, int r_max, int64_t *offs);
cudaError_t launch_encode(const uint16_t *k, const uint16_t *v, const int64_t *tok0, const int32_t *blen,
                          const int64_t *offs, uint16_t *arena, int32_t *rank_k, int32_t *rank_v, float *sigma,
                          float *vt, int32_t *status, int nb, int hkv, int d, int r_min, int r_max,
                          int64_t budget_k, int64_t budget_v, cudaStream_t stream);

// INT8 storage of a packed arena (milo_int8.cu): `groups` 128-byte cores,
// 64 codes and one parameter word each.
cudaError_t launch_quant_int8(const void *packed, int64_t groups, void *codes, void *params, cudaStream_t stream);
cudaError_t launch_dequant_int8(const void *codes, const void *params, int64_t groups, void *packed,
                                cudaStream_t stream);
// The same for a plan's arena, with the padding of every factor read back as 0.
// max_factor_groups: the most 8x8 cores of one factor (C^K, P^K, C^V or P^V).
cudaError_t launch_dequant_plan_int8(const EntryDev *entries, int num_entries, int head_dim, int64_t max_factor_groups,
                                     const void *codes, const void *params, void *packed, cudaStream_t stream);

// Fixed scratch of milo_attn_decode_static (a file-scope device array).
constexpr size_t kStaticWorkspaceBytes = size_t(8) << 20;
// Device address of that array on the current device (looked up once per
// device).
cudaError_t static_workspace(void **ptr);

}  // namespace milo
