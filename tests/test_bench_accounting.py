"""The benchmark's accounting (tokens attended, algorithmic bytes and FLOPs
of one decode call), which every roofline fraction divides by, checked
against a count taken from the tensors and the loops of the attention
itself on small layers (CPU only)."""
import numpy as np
import pytest

import bench
from paper_2609_29913_gb300 import workloads as W


def counted(layer):
    """Bytes: every factor at its true rank as stored (bf16), the tails, q
    and the fp32 output.  FLOPs (a multiply-add is 2): the products of the
    rank-space attention loop by loop."""
    hk, d, G = layer.num_kv_heads, layer.head_dim, layer.num_q_heads // layer.num_kv_heads
    nbytes = 0
    flops = 0
    for e in range(len(layer.rank_k)):
        n = int(layer.block_len[e // hk])
        rk, rv = int(layer.rank_k[e]), int(layer.rank_v[e])
        nbytes += 2 * (n * rk + rk * d + n * rv + rv * d)       # C^K, P^K, C^V, P^V in bf16
        per_row = 0
        per_row += 2 * rk * d      # q~ = P^K q
        per_row += 2 * n * rk      # s = C^K q~
        per_row += 2 * n * rv      # v~ = sum_t p_t C^V_t
        per_row += 2 * rv * d      # o = P^V^T v~
        flops += per_row * layer.batch * G
    T = np.diff(layer.tail_offsets)
    for i in range(layer.batch):
        nbytes += int(T[i]) * hk * d * 2 * 2                    # K and V rows of the tail
        flops += int(T[i]) * hk * G * (2 * d + 2 * d)           # scores and values per tail token
    nbytes += layer.batch * layer.num_q_heads * d * 2          # q (bf16)
    nbytes += layer.batch * layer.num_q_heads * d * 4          # out (fp32)
    tokens = layer.batch * int(np.sum(layer.block_len)) + int(T.sum())
    return tokens, nbytes, flops


@pytest.mark.parametrize("shape", [
    (28, 4, 128, [512, 300, 7], (0, 13, 64, 128), 3, [5, 0, 70]),
    (14, 2, 64, [256, 1], (8, 16, 32), 1, [0]),
    (40, 8, 128, [64], (1, 128), 2, [513, 2]),
])
def test_layer_totals_match_a_count(shape):
    hq, hkv, d, bl, ranks, batch, tails = shape
    layer = W.make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                               rank_choices=ranks, batch=batch, tail_lengths=tails, seed=3)
    got = bench.layer_totals(hq, hkv, d, layer.block_len, layer.rank_k, layer.rank_v,
                             np.diff(layer.tail_offsets), batch)
    assert got == counted(layer)


def test_workload_totals_sum_the_layers():
    """workload_totals (from the rank and tail tables alone) equals the sum
    of layer_totals over the layers actually generated (2k workload)."""
    cfg = W.by_name("qwen0.5b-1L-2k")
    tot = bench.workload_totals(cfg, W)
    want = [0, 0, 0]
    for l in range(cfg.layers):
        layer = W.make_config_layer(cfg, l, device="cpu")
        t = counted(layer)
        want = [a + b for a, b in zip(want, t)]
    assert list(tot) == want
