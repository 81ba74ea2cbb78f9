/* A plain C caller of libmilo's host-only entry points (no GPU needed):
 * proves the header compiles as C and the ABI is callable without Python.
 * Prints one line per result; tests/test_c_abi.py compares them with the
 * ctypes binding. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "milo.h"

int main(void)
{
    /* two blocks (33 and 512 tokens) x 2 KV heads, head_dim 64, ranks below */
    const int32_t block_len[2] = {33, 512};
    const int32_t rank_k[4] = {8, 13, 64, 0};
    const int32_t rank_v[4] = {5, 16, 32, 64};
    int64_t off[4][4];
    int64_t cur = 0;
    for (int e = 0; e < 4; ++e) {
        const int64_t n = block_len[e / 2];
        const int64_t sz[4] = {n * rank_k[e], (int64_t)rank_k[e] * 64, n * rank_v[e], (int64_t)rank_v[e] * 64};
        for (int f = 0; f < 4; ++f) {
            off[f][e] = cur;
            cur += (sz[f] + 7) / 8 * 8;
        }
    }
    static uint16_t arena[1 << 17];
    if (cur > (int64_t)(sizeof arena / 2)) return 2;
    milo_block_table_t t;
    memset(&t, 0, sizeof t);
    t.num_blocks = 2;
    t.num_kv_heads = 2;
    t.head_dim = 64;
    t.block_len = block_len;
    t.rank_k = rank_k;
    t.rank_v = rank_v;
    t.off_ck = off[0];
    t.off_pk = off[1];
    t.off_cv = off[2];
    t.off_pv = off[3];
    t.arena = arena;
    t.arena_elems = cur;

    printf("version %d\n", (int)milo_version());
    printf("validate %d\n", (int)milo_validate_table(&t));
    int64_t packed[16], total = 0;
    printf("layout %d\n", (int)milo_packed_layout(&t, packed, &total));
    printf("packed_total %lld\n", (long long)total);
    int32_t nchunks = 0;
    printf("chunks_status %d\n", (int)milo_chunk_prefix(&t, 0, NULL, NULL, NULL, &nchunks));
    printf("chunks %d\n", (int)nchunks);
    int32_t nseg = 0, nslot = 0;
    printf("partition_status %d\n", (int)milo_partition_prefix(&t, 3, 0, NULL, NULL, NULL, NULL, NULL, &nseg, &nslot));
    printf("segments %d\n", (int)nseg);
    printf("slots %d\n", (int)nslot);

    /* a rank above head_dim is a bad table; an odd offset an alignment error */
    int32_t bad_rank[4] = {8, 13, 65, 0};
    t.rank_k = bad_rank;
    printf("bad_rank %d\n", (int)milo_validate_table(&t));
    t.rank_k = rank_k;
    int64_t odd[4] = {off[0][0] + 1, off[0][1], off[0][2], off[0][3]};
    t.off_ck = odd;
    printf("odd_offset %d\n", (int)milo_validate_table(&t));
    printf("status_string %s\n", milo_status_string(MILO_ERR_BAD_TABLE));
    printf("null_plan %d\n", (int)milo_prefix_set_tensor_min_rows(NULL, 4));
    return 0;
}
