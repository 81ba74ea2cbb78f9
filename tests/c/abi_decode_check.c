/* A plain C caller of the whole decode path on the GPU, with no Python on
 * it: builds a seeded random block table in host memory, copies it to the
 * device with the CUDA runtime, builds a plan, runs milo_attn_decode (with a
 * workspace) and milo_attn_decode_static, and writes the inputs and both
 * outputs to files in the directory given as argv[1], where
 * tests/test_gpu_c_abi.py compares them with the oracle.  The generator draws
 * bf16 bit patterns only (no arithmetic of the method). */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "milo.h"

enum { NB = 3, HKV = 2, G = 7, HQ = HKV * G, D = 128, BATCH = 2 };

static uint64_t rng = 0x9E3779B97F4A7C15ull;
static uint32_t next32(void)
{
    rng ^= rng << 13;
    rng ^= rng >> 7;
    rng ^= rng << 17;
    return (uint32_t)(rng >> 32);
}
/* a bf16 of magnitude in [2^-4, 2) and random sign */
static uint16_t draw_bf16(void)
{
    const uint32_t r = next32();
    const uint32_t exp = 123 + (r >> 8) % 5, mant = r & 0x7F, sign = (r >> 20) & 1;
    return (uint16_t)((sign << 15) | (exp << 7) | mant);
}

static int write_file(const char *dir, const char *name, const void *p, size_t bytes)
{
    char path[4096];
    snprintf(path, sizeof path, "%s/%s", dir, name);
    FILE *f = fopen(path, "wb");
    if (!f) return 1;
    const size_t w = fwrite(p, 1, bytes, f);
    fclose(f);
    return w == bytes ? 0 : 1;
}

#define CHECK_CUDA(x)                                                          \
    do {                                                                       \
        cudaError_t e_ = (x);                                                  \
        if (e_ != cudaSuccess) {                                               \
            fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));           \
            return 10;                                                         \
        }                                                                      \
    } while (0)
#define CHECK_MILO(x)                                                          \
    do {                                                                       \
        milo_status_t s_ = (x);                                                \
        if (s_ != MILO_OK) {                                                   \
            fprintf(stderr, "%s: %s (%s)\n", #x, milo_status_string(s_),       \
                    milo_last_error_message());                                \
            return 20;                                                         \
        }                                                                      \
    } while (0)

int main(int argc, char **argv)
{
    if (argc < 2) return 1;
    const int32_t block_len[NB] = {512, 129, 40};
    int32_t rank_k[NB * HKV], rank_v[NB * HKV];
    const int32_t choices[6] = {0, 7, 16, 33, 64, 128};
    for (int e = 0; e < NB * HKV; ++e) {
        rank_k[e] = choices[next32() % 6];
        rank_v[e] = choices[next32() % 6];
    }
    int64_t off[4][NB * HKV];
    int64_t elems = 0;
    for (int e = 0; e < NB * HKV; ++e) {
        const int64_t n = block_len[e / HKV];
        const int64_t sz[4] = {n * rank_k[e], (int64_t)rank_k[e] * D, n * rank_v[e], (int64_t)rank_v[e] * D};
        for (int f = 0; f < 4; ++f) {
            off[f][e] = elems;
            elems += (sz[f] + 7) / 8 * 8;
        }
    }
    uint16_t *arena = calloc((size_t)elems + 8, 2);
    for (int64_t i = 0; i < elems; ++i) arena[i] = draw_bf16();
    const int64_t tail_offsets[BATCH + 1] = {0, 70, 70 + 200};
    const int64_t tail_rows = tail_offsets[BATCH];
    uint16_t *q = malloc((size_t)BATCH * HQ * D * 2);
    uint16_t *tk = malloc((size_t)tail_rows * HKV * D * 2), *tv = malloc((size_t)tail_rows * HKV * D * 2);
    for (int i = 0; i < BATCH * HQ * D; ++i) q[i] = draw_bf16();
    for (int64_t i = 0; i < tail_rows * HKV * D; ++i) {
        tk[i] = draw_bf16();
        tv[i] = draw_bf16();
    }

    void *d_arena, *d_q, *d_tk, *d_tv, *d_toff, *d_out, *d_out2, *d_ws;
    CHECK_CUDA(cudaMalloc(&d_arena, (size_t)elems * 2 + 16));
    CHECK_CUDA(cudaMemcpy(d_arena, arena, (size_t)elems * 2, cudaMemcpyHostToDevice));
    milo_block_table_t t;
    memset(&t, 0, sizeof t);
    t.num_blocks = NB;
    t.num_kv_heads = HKV;
    t.head_dim = D;
    t.block_len = block_len;
    t.rank_k = rank_k;
    t.rank_v = rank_v;
    t.off_ck = off[0];
    t.off_pk = off[1];
    t.off_cv = off[2];
    t.off_pv = off[3];
    t.arena = d_arena;
    t.arena_elems = elems;
    cudaStream_t stream;
    CHECK_CUDA(cudaStreamCreate(&stream));
    milo_prefix_t *plan = NULL;
    CHECK_MILO(milo_prefix_create(&t, HQ, BATCH, stream, &plan));
    CHECK_CUDA(cudaFree(d_arena));  /* the plan holds its own packed copy */

    CHECK_CUDA(cudaMalloc(&d_q, (size_t)BATCH * HQ * D * 2));
    CHECK_CUDA(cudaMalloc(&d_tk, (size_t)tail_rows * HKV * D * 2));
    CHECK_CUDA(cudaMalloc(&d_tv, (size_t)tail_rows * HKV * D * 2));
    CHECK_CUDA(cudaMalloc(&d_toff, sizeof tail_offsets));
    CHECK_CUDA(cudaMalloc(&d_out, (size_t)BATCH * HQ * D * 4));
    CHECK_CUDA(cudaMalloc(&d_out2, (size_t)BATCH * HQ * D * 4));
    CHECK_CUDA(cudaMemcpy(d_q, q, (size_t)BATCH * HQ * D * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(d_tk, tk, (size_t)tail_rows * HKV * D * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(d_tv, tv, (size_t)tail_rows * HKV * D * 2, cudaMemcpyHostToDevice));
    CHECK_CUDA(cudaMemcpy(d_toff, tail_offsets, sizeof tail_offsets, cudaMemcpyHostToDevice));
    size_t ws_bytes = 0;
    CHECK_MILO(milo_workspace_size(plan, BATCH, 200, &ws_bytes));
    CHECK_CUDA(cudaMalloc(&d_ws, ws_bytes));
    CHECK_MILO(milo_attn_decode(plan, d_q, BATCH, d_tk, d_tv, d_toff, tail_rows, 200, 0.f, d_out, d_ws, ws_bytes,
                                stream));
    CHECK_MILO(milo_attn_decode_static(plan, d_q, BATCH, d_tk, d_tv, d_toff, tail_rows, 200, 0.f, d_out2, stream));
    CHECK_CUDA(cudaStreamSynchronize(stream));
    int32_t code = -1;
    CHECK_MILO(milo_get_device_status(plan, stream, 0, &code));
    if (code != 0) {
        fprintf(stderr, "device status %d\n", (int)code);
        return 30;
    }
    float *out = malloc((size_t)BATCH * HQ * D * 4), *out2 = malloc((size_t)BATCH * HQ * D * 4);
    CHECK_CUDA(cudaMemcpy(out, d_out, (size_t)BATCH * HQ * D * 4, cudaMemcpyDeviceToHost));
    CHECK_CUDA(cudaMemcpy(out2, d_out2, (size_t)BATCH * HQ * D * 4, cudaMemcpyDeviceToHost));
    milo_call_info_t info;
    CHECK_MILO(milo_call_info(plan, BATCH, 200, &info));
    CHECK_MILO(milo_prefix_destroy(plan));

    const char *dir = argv[1];
    int bad = 0;
    bad |= write_file(dir, "block_len.i32", block_len, sizeof block_len);
    bad |= write_file(dir, "rank_k.i32", rank_k, sizeof rank_k);
    bad |= write_file(dir, "rank_v.i32", rank_v, sizeof rank_v);
    bad |= write_file(dir, "off.i64", off, sizeof off);
    bad |= write_file(dir, "arena.u16", arena, (size_t)elems * 2);
    bad |= write_file(dir, "q.u16", q, (size_t)BATCH * HQ * D * 2);
    bad |= write_file(dir, "tail_k.u16", tk, (size_t)tail_rows * HKV * D * 2);
    bad |= write_file(dir, "tail_v.u16", tv, (size_t)tail_rows * HKV * D * 2);
    bad |= write_file(dir, "tail_offsets.i64", tail_offsets, sizeof tail_offsets);
    bad |= write_file(dir, "out.f32", out, (size_t)BATCH * HQ * D * 4);
    bad |= write_file(dir, "out_static.f32", out2, (size_t)BATCH * HQ * D * 4);
    printf("path %d kernels %d\n", (int)info.path, (int)info.kernels);
    return bad ? 40 : 0;
}
