"""GPU parity: libmilo's CUDA path against the fp64 oracle, through the C ABI.

Tolerances (fp32 output of bf16 inputs): max-abs 1e-2 and relative L2 2e-3
over each compared output tensor.  Index and layout handling (packing) is
checked bit-exactly."""
import math
import zlib

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

ATOL = 1e-2
RTOL_L2 = 2e-3


@pytest.fixture(scope="module")
def env(oracle):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_29913_gb300 import build, milo, workloads
    build.build()
    milo.lib()
    return dict(milo=milo, W=workloads, oracle=oracle)


def decode(env, layer, scale=0.0, max_tail=None, plan=None, out=None, workspace=None):
    milo = env["milo"]
    pre = plan or milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max()) if layer.batch else 0
    if max_tail is not None:
        mt = max_tail
    res = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt, scale, out=out,
                     workspace=workspace)
    torch.cuda.synchronize()
    assert pre.status(clear=True) == 0, "device status word set"
    return res, pre


def compare(got, ref, what=""):
    got = np.asarray(got, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = np.abs(got - ref).max()
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    assert err <= ATOL and rel <= RTOL_L2, f"{what}: max-abs {err:.3e} rel-L2 {rel:.3e}"
    return err, rel


CASES = {
    # name: (hq, hkv, d, block_lens, rank_choices, batch, tail_lengths, separate_kv)
    "cfg0-shape": (14, 2, 64, [256] * 8, (8, 16, 32), 1, None, False),
    "ragged-d128": (7, 1, 128, [1, 7, 129, 64, 200], (1, 4, 7, 8, 13, 64, 128), 1, [65], True),
    "gqa7-b2": (28, 4, 128, [512, 512, 100], (16, 32, 64, 96, 128), 2, [0, 130], False),
    "d64-b3": (8, 1, 64, [33, 100, 9], (5, 64, 0), 3, [1, 64, 0], True),
    "gqa5-long-tail": (40, 8, 128, [300, 512], (32, 41, 77, 128), 2, [1029, 17], True),
    "g16": (16, 1, 128, [64, 65], (128, 3), 1, [10], True),
    "g32-d64": (32, 1, 64, [100], (20,), 1, [70], False),
    "tail-only": (14, 2, 64, [], (8,), 2, [5, 300], False),
    "batch64-multipass": (28, 4, 128, [128, 64], (16, 128, 40), 64, [33] * 64, True),
    "batch9-odd-groups": (21, 3, 64, [96, 40], (7, 64), 9, list(range(1, 10)), True),
    # 21 rows per KV head: 3 row groups (two-group blocks, the last half
    # empty) and 9 tail items (two to a block, the last alone), at d = 128
    "d128-odd-row-groups": (21, 3, 128, [512, 77, 300], (16, 64, 96, 128), 3, [5, 60, 1], True),
    "rank0": (4, 2, 64, [50, 70], (0,), 1, [3], True),
    # G = 10 at batch 2 (20 rows, chunk grid): tail items of 8 and 2 rows
    "g10-b2": (20, 2, 128, [130, 512, 7], (8, 64, 128), 2, [70, 129], True),
    # G = 12 at batch 3 (36 rows: the tensor-core grid) with long tail items
    # of 8 and 4 rows
    "g12-b3-tensor": (24, 2, 64, [256, 300], (16, 33, 64), 3, [600, 0, 65], True),
    # G = 12 without a prefix: a chunk grid of tail items alone
    "g12-tail-only": (12, 1, 128, [], (8,), 2, [1, 200], False),
}


def test_rank0_entries_mixed_with_others_d128(env):
    """Entries of rank 0 in K and V, in K only and in V only, between entries
    of rank 16 and 128, in one plan at head dimension 128 (an entry of rank 0
    in both has no coefficient rows: its chunk's piece copies nothing)."""
    W = env["W"]
    #          block:  0        1        2         3        4
    rk = np.array([[0, 16], [0, 128], [16, 0], [128, 0], [0, 0]], dtype=np.int32)
    rv = np.array([[0, 0], [128, 0], [0, 16], [0, 128], [16, 0]], dtype=np.int32)
    layer = W.build_layer(14, 2, 128, [40, 512, 96, 300, 33], rk, rv, batch=2, tail_lengths=[17, 70],
                          seed=12, device="cuda")
    out, pre = decode(env, layer)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(out.cpu().numpy(), ref, "rank0 mixed d128")
    pre.close()


@pytest.mark.parametrize("name", sorted(CASES))
def test_small_cases_match_oracle(env, name):
    hq, hkv, d, bl, ranks, batch, tails, sep = CASES[name]
    layer = env["W"].make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                                      rank_choices=ranks, batch=batch, tail_lengths=tails,
                                      seed=zlib.crc32(name.encode()) % 1000, device="cuda",
                                      separate_kv_ranks=sep)
    out, pre = decode(env, layer)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(out.cpu().numpy(), ref, name)
    pre.close()


@pytest.mark.parametrize("batch", [1, 5])
def test_longest_block(env, batch):
    """A block of 65536 tokens (the longest a table accepts) at ranks 128 and
    16 beside a 3-token block, at batch 1 (7 rows: the chunk grid, the long
    entry cut into chunks of at most 1024 tokens) and batch 5 (35 rows: the
    tensor-core grid, the entry cut at 32-token boundaries over the shares)."""
    milo, W = env["milo"], env["W"]
    layer = W.build_layer(7, 1, 128, [65536, 3], [[128], [8]], [[16], [5]], batch=batch,
                          tail_lengths=[70 + 3 * i for i in range(batch)], seed=65, device="cuda")
    out, pre = decode(env, layer)
    mt = int(np.diff(layer.tail_offsets).max())
    assert milo.milo_call_info(pre.plan, batch, mt)["path"] == (0 if batch == 1 else 1)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(out.cpu().numpy(), ref, f"longest block, batch {batch}")
    pre.close()


def test_peaked_softmax(env):
    layer = env["W"].make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128,
                                      block_lens=[512, 77, 512], rank_choices=(16, 64, 128),
                                      batch=2, tail_lengths=[40, 200], seed=3, device="cuda",
                                      q_scale=30.0)
    out, _ = decode(env, layer)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(out.cpu().numpy(), ref, "peaked")


def test_outlier_maximum_takes_the_record_path(env):
    """Scores of a few late tokens 256 times larger than the rest.  Every
    prefix chunk fixes its KV head's shared reference maximum (if it is the
    first) from the scores of its first piece, which here are ordinary
    (tokens 0-255 at rank 16), so the chunk holding tokens 300-309 ends with a
    maximum hundreds above the reference whichever item set it: its result
    must go through the listed-record merge rather than the accumulators."""
    W = env["W"]
    layer = W.build_layer(14, 2, 128, [1024, 512], [[16, 16], [64, 32]], batch=1, tail_lengths=[70],
                          seed=8, device="cuda")
    A = layer.arena
    for e in range(2):  # block 0, both KV heads
        r = int(layer.rank_k[e])
        off = int(layer.off_ck[e])
        A[off + 300 * r:off + 310 * r] *= 256.0
    out, pre = decode(env, layer)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(out.cpu().numpy(), ref, "outlier")
    out2, _ = decode(env, layer, plan=pre)  # the accumulators were cleared
    compare(out2.cpu().numpy(), ref, "outlier again")
    pre.close()


@pytest.mark.parametrize("batch,hot_tail", [(3, False), (3, True), (10, True)])
def test_outlier_maximum_batched_row_groups(env, batch, hot_tail):
    """The listed-record merge with several row groups of 8 query rows: GQA 7,
    so most queries' rows straddle two row groups, whose finish warps both
    read such an item's record.  Prefix tokens 300-309 of every KV head get
    scores 256 times larger; with hot_tail, query 1's tail keys are scaled
    the same way, so tail items (one per query) take the record path too."""
    W = env["W"]
    tails = [70 + 13 * i for i in range(batch)]
    layer = W.build_layer(14, 2, 128, [1024, 512], [[16, 16], [64, 32]], batch=batch, tail_lengths=tails,
                          seed=18 + batch, device="cuda")
    A = layer.arena
    for e in range(2):
        r = int(layer.rank_k[e])
        off = int(layer.off_ck[e])
        A[off + 300 * r:off + 310 * r] *= 256.0
    if hot_tail:
        o0, o1 = int(layer.tail_offsets[1]), int(layer.tail_offsets[2])
        layer.tail_k[o0:o1] *= 64.0
    out, pre = decode(env, layer)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(out.cpu().numpy(), ref, "batched outlier")
    out2, _ = decode(env, layer, plan=pre)  # the accumulators and lists were cleared
    compare(out2.cpu().numpy(), ref, "batched outlier again")
    pre.close()


def test_explicit_scale(env):
    layer = env["W"].make_random_case(num_q_heads=7, num_kv_heads=1, head_dim=64,
                                      block_lens=[128, 64], rank_choices=(16, 40),
                                      batch=1, tail_lengths=[20], seed=4, device="cuda")
    out, _ = decode(env, layer, scale=0.3)
    ref = env["oracle"].attention(**layer.to_numpy_bits(), scale=0.3)
    compare(out.cpu().numpy(), ref, "scale")


def test_nan_poisoned_gaps_do_not_leak(env):
    layer = env["W"].make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=64,
                                      block_lens=[33, 70, 129], rank_choices=(3, 5, 13),
                                      batch=1, tail_lengths=[9], seed=5, device="cuda",
                                      poison_gaps=True)
    assert torch.isnan(layer.arena.float()).any()
    out, _ = decode(env, layer)
    bits = layer.to_numpy_bits()
    ref = env["oracle"].attention(**bits)
    compare(out.cpu().numpy(), ref, "poisoned")


def test_identity_basis_equals_dense_attention(env):
    """P = first r rows of the identity (exact in bf16): the compressed
    attention equals plain dense attention over K = [C, 0], V = [C, 0]."""
    W = env["W"]
    d, n, hkv, hq = 64, 96, 1, 4
    layer = W.build_layer(hq, hkv, d, [n, n], [[48], [64]], batch=1, tail_lengths=[0],
                          seed=6, device="cuda", basis="identity")
    out, _ = decode(env, layer)
    A = layer.arena.float()
    keys, vals = [], []
    for b in range(2):
        r = int(layer.rank_k[b])
        C = A[int(layer.off_ck[b]):int(layer.off_ck[b]) + n * r].view(n, r)
        Cv = A[int(layer.off_cv[b]):int(layer.off_cv[b]) + n * r].view(n, r)
        keys.append(torch.nn.functional.pad(C, (0, d - r)))
        vals.append(torch.nn.functional.pad(Cv, (0, d - r)))
    K, V = torch.cat(keys), torch.cat(vals)
    q = layer.q.float()[0]
    ref = torch.softmax(q @ K.T / math.sqrt(d), dim=-1) @ V
    err = (out[0] - ref).abs().max().item()
    assert err < 2e-5, err


def test_packed_arena_is_bit_exact(env):
    """Download the packed arena and undo the documented layout in numpy."""
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=8, num_kv_heads=2, head_dim=64,
                               block_lens=[5, 64, 130], rank_choices=(1, 7, 8, 13, 64),
                               batch=1, tail_lengths=[0], seed=7, device="cuda")
    table = milo.HostTable.from_layer(layer)
    pre = milo.Prefix(table, 8, 1)
    offs, total = milo.milo_packed_layout(table)
    info = pre.info
    assert info["packed_bytes"] == total
    class _View:  # a view of the plan's packed arena (device pointer, no copy)
        __cuda_array_interface__ = dict(shape=(total,), typestr="|u1",
                                        data=(info["packed_arena"], False), version=3)
    packed = torch.as_tensor(_View(), device="cuda")
    torch.cuda.synchronize()
    pk = packed.cpu().numpy().view(np.uint16)
    logical = layer.to_numpy_bits()["arena"]
    d = 64
    for e in range(len(layer.rank_k)):
        n = int(layer.block_len[e // 2])
        for f, (r, loff) in enumerate(((layer.rank_k[e], layer.off_ck[e]), (layer.rank_k[e], layer.off_pk[e]),
                                       (layer.rank_v[e], layer.off_cv[e]), (layer.rank_v[e], layer.off_pv[e]))):
            r = int(r)
            r8 = (r + 7) // 8 * 8
            base = int(offs[e, f]) // 2
            if f % 2 == 0:   # C: [token group][rank group] 8x8 tiles over the whole entry
                n8 = (n + 7) // 8 * 8
                full = np.zeros((n8, r8), np.uint16)
                full[:n, :r] = logical[loff:loff + n * r].reshape(n, r)
                got = np.zeros_like(full)
                for tg in range(n8 // 8):
                    for rg in range(r8 // 8):
                        o = base + (tg * (r8 // 8) + rg) * 64
                        got[8 * tg: 8 * tg + 8, 8 * rg: 8 * rg + 8] = pk[o:o + 64].reshape(8, 8)
            else:            # P: [rank group][column group] 8x8 tiles
                full = np.zeros((r8, d), np.uint16)
                full[:r] = logical[loff:loff + r * d].reshape(r, d)
                got = np.zeros_like(full)
                for jg in range(r8 // 8):
                    for cg in range(d // 8):
                        o = base + (jg * (d // 8) + cg) * 64
                        got[8 * jg: 8 * jg + 8, 8 * cg: 8 * cg + 8] = pk[o:o + 64].reshape(8, 8)
            np.testing.assert_array_equal(got, full, err_msg=f"entry {e} factor {f}")
    pre.close()


def test_repeated_calls_batches_and_graph_capture(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128,
                               block_lens=[512, 256, 99], rank_choices=(16, 64, 128),
                               batch=4, tail_lengths=[10, 0, 64, 129], seed=8, device="cuda")
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    pre = milo.Prefix.from_layer(layer, max_batch=4)
    first, _ = decode(env, layer, plan=pre)
    compare(first.cpu().numpy(), ref, "repeat")
    # Items add their scaled partial sums into fp32 accumulators with atomics
    # in whatever order they finish, so repeated calls agree to fp32 rounding,
    # not bit for bit: each output is a sum of some tens of partials, each
    # addition rounding at 2^-24 of the running sum, and the running sums of
    # signed values can exceed the final one several times over.
    rep_tol = 2e-5 * first.abs().max().item()
    for _ in range(3):
        again, _ = decode(env, layer, plan=pre)
        assert (again - first).abs().max().item() <= rep_tol
    # a smaller batch on the same plan (queries 0..1)
    sub = W.LayerInputs(layer.num_q_heads, layer.num_kv_heads, layer.head_dim, layer.block_len,
                        layer.rank_k, layer.rank_v, layer.off_ck, layer.off_pk, layer.off_cv,
                        layer.off_pv, layer.arena, layer.q[:2].contiguous(), layer.tail_k,
                        layer.tail_v, layer.tail_offsets[:3])
    o2, _ = decode(env, sub, plan=pre)
    compare(o2.cpu().numpy(), ref[:2], "sub-batch")
    # CUDA graph of three calls
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    out = torch.empty_like(first)
    ws = torch.empty(pre.workspace_size(4, 129), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, 129, out=out, workspace=ws, stream=s)
        s.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            for _ in range(3):
                pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, 129, out=out, workspace=ws,
                           stream=s)
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert (out - first).abs().max().item() <= rep_tol
    assert pre.status() == 0
    pre.close()


def test_canaries_around_out_and_workspace(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=64,
                               block_lens=[256, 100], rank_choices=(8, 32),
                               batch=2, tail_lengths=[5, 70], seed=9, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    n = layer.batch * 14 * 64
    big = torch.full((n + 2048,), 12345.0, device="cuda")
    out = big[1024:1024 + n].view(layer.batch, 14, 64)
    need = pre.workspace_size(layer.batch, 70)
    wbig = torch.full((need + 8192,), 77, dtype=torch.uint8, device="cuda")
    ws = wbig[4096:4096 + need]
    decode(env, layer, plan=pre, out=out, workspace=ws)
    assert (big[:1024] == 12345.0).all() and (big[1024 + n:] == 12345.0).all()
    assert (wbig[:4096] == 77).all() and (wbig[4096 + need:] == 77).all()
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), "canary")


def test_argument_errors_are_reported(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=4, num_kv_heads=1, head_dim=64, block_lens=[16],
                               rank_choices=(8,), batch=1, tail_lengths=[0], seed=10, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    out = torch.empty((1, 4, 64), device="cuda")
    ws = torch.empty(pre.workspace_size(1, 0), dtype=torch.uint8, device="cuda")
    with pytest.raises(milo.MiloError) as ei:
        milo.milo_attn_decode(pre.plan, layer.q.data_ptr(), 2, 0, 0, 0, 0, 0, 0.0, out.data_ptr(),
                              ws.data_ptr(), ws.numel())
    assert ei.value.status == 1          # batch above max_batch
    with pytest.raises(milo.MiloError) as ei:
        milo.milo_attn_decode(pre.plan, layer.q.data_ptr(), 1, 0, 0, 0, 0, 0, 0.0, out.data_ptr(),
                              ws.data_ptr(), 16)
    assert ei.value.status == 8          # workspace too small
    with pytest.raises(milo.MiloError) as ei:
        milo.milo_attn_decode(pre.plan, layer.q.data_ptr(), 1, 0, 0, 0, 0, 5, 0.0, out.data_ptr(),
                              ws.data_ptr(), ws.numel())
    assert ei.value.status == 1          # tail promised but no tail pointers
    pre.close()


def test_tail_longer_than_promised_sets_status(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=4, num_kv_heads=1, head_dim=64, block_lens=[16],
                               rank_choices=(8,), batch=1, tail_lengths=[200], seed=11, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, 64)
    torch.cuda.synchronize()
    assert pre.status(clear=True) == 7   # MILO_ERR_DEVICE_BOUNDS
    assert pre.status() == 0
    pre.close()


# ---------------------------------------------------------------- full size
def oracle_subset(env, layer, queries, g):
    """Oracle on the rows of KV head g for the given queries (exact subset)."""
    bits = layer.to_numpy_bits()
    hkv = layer.num_kv_heads
    G = layer.num_q_heads // hkv
    ent = np.arange(layer.num_blocks) * hkv + g
    q = bits["q"][queries][:, g * G:(g + 1) * G]
    args = dict(num_kv_heads=1, head_dim=layer.head_dim, block_len=layer.block_len,
                rank_k=layer.rank_k[ent], rank_v=layer.rank_v[ent], off_ck=layer.off_ck[ent],
                off_pk=layer.off_pk[ent], off_cv=layer.off_cv[ent], off_pv=layer.off_pv[ent],
                arena=bits["arena"], q=np.ascontiguousarray(q))
    if "tail_k" in bits:
        tk, tv, toff = [], [], [0]
        for i in queries:
            a, b = layer.tail_offsets[i], layer.tail_offsets[i + 1]
            tk.append(bits["tail_k"][a:b, g:g + 1])
            tv.append(bits["tail_v"][a:b, g:g + 1])
            toff.append(toff[-1] + b - a)
        args.update(tail_k=np.ascontiguousarray(np.concatenate(tk)),
                    tail_v=np.ascontiguousarray(np.concatenate(tv)), tail_offsets=np.array(toff))
    return env["oracle"].attention(**args)


def test_qwen05b_one_layer_full(env):
    W = env["W"]
    layer = W.make_config_layer(W.by_name("qwen0.5b-1L-2k"), 0, device="cuda")
    out, _ = decode(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), "qwen0.5b-1L-2k")


@pytest.mark.parametrize("layer_idx", [0, 27])
def test_qwen7b_batch1_layers_full(env, layer_idx):
    W = env["W"]
    layer = W.make_config_layer(W.by_name("qwen7b-28L-32k-b1"), layer_idx, device="cuda")
    out, _ = decode(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), f"qwen7b-28L-32k-b1 L{layer_idx}")


def worst_row_rel_l2(got, ref):
    """The largest relative L2 error over the (query, head) rows."""
    d = got.shape[-1]
    g = np.asarray(got, np.float64).reshape(-1, d)
    r = np.asarray(ref, np.float64).reshape(-1, d)
    return float((np.linalg.norm(g - r, axis=1) / np.maximum(np.linalg.norm(r, axis=1), 1e-30)).max())


@pytest.mark.parametrize("name", ["qwen7b-28L-32k-b64", "qwen14b-48L-128k-b16", "qwen7b-1L-1M-b8"])
def test_batched_workloads_whole_layer(env, name):
    """Layer 0 of each batched workload against the oracle over the whole
    output tensor [batch, Hq, d] (every query, every head)."""
    W = env["W"]
    layer = W.make_config_layer(W.by_name(name), 0, device="cuda")
    out, pre = decode(env, layer)
    got = out.cpu().numpy()
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    err, rel = compare(got, ref, f"{name} layer 0")
    print(f"{name} layer 0: max-abs {err:.3e} rel-L2 {rel:.3e} "
          f"worst (query, head) rel-L2 {worst_row_rel_l2(got, ref):.3e}")
    pre.close()


@pytest.mark.parametrize("name,queries,heads", [("qwen7b-28L-32k-b64", [0, 63], [0, 3]),
                                                ("qwen14b-48L-128k-b16", [0, 15], [0, 7])])
def test_batched_workloads_last_layer_sampled(env, name, queries, heads):
    """The last layer of the multi-layer batched workloads on a few (query,
    KV head) subsets, each an exact subproblem the oracle solves alone."""
    W = env["W"]
    cfg = W.by_name(name)
    layer = W.make_config_layer(cfg, cfg.layers - 1, device="cuda")
    out, _ = decode(env, layer)
    G = layer.num_q_heads // layer.num_kv_heads
    o = out.cpu().numpy()
    assert np.isfinite(o).all()
    for g in heads:
        ref = oracle_subset(env, layer, queries, g)
        compare(o[queries][:, g * G:(g + 1) * G], ref, f"{name} g{g}")


def test_bounded_wait_runs_out_and_reports(env):
    """The bounded mbarrier wait of the kernels, on a barrier nothing
    completes (a 50 ms limit): the status word reads MILO_ERR_TIMEOUT, the
    kernel ends, and the same plan then decodes correctly.  A wait on a
    completed barrier reports nothing."""
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128, block_lens=[256, 64],
                               rank_choices=(16, 64), batch=2, tail_lengths=[10, 30], seed=5, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    assert pre.status(clear=True) == 0
    milo.milo_check_bounded_wait(pre.plan, 50_000_000, True)
    assert pre.status() == 0
    milo.milo_check_bounded_wait(pre.plan, 50_000_000, False)
    assert pre.status(clear=True) == 6  # MILO_ERR_TIMEOUT
    assert pre.status() == 0
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    out = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, 30)
    torch.cuda.synchronize()
    assert pre.status() == 0
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    got = out.cpu().numpy().astype(np.float64)
    assert np.abs(got - ref).max() <= 1e-2
    with pytest.raises(milo.MiloError):
        milo.milo_check_bounded_wait(pre.plan, 10, False)
    pre.close()
