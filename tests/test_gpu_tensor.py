"""GPU parity of the tensor-core path (calls with at least
milo_tensor_min_rows() query rows per KV head) against the fp64 oracle,
through the C ABI.  (Its cases with more than 8 query heads per KV head,
G = 12 and 32, sit in test_gpu_parity.py.)

The cases put the row count at the path's threshold and across a 128-row
tile boundary, run calls of one tile of at most 64 rows (spread 16 per
tensor-memory lane quarter) and fuller ones, and cover head dimensions 64 and 128, ragged blocks, ranks 0
(K, V or both) next to full ranks, separate K and V ranks, a peaked softmax,
late outlier scores that force the listed-record merge, calls without tails,
shares that cross KV heads, and repeated and graph-captured calls.
Tolerances as in the other parity tests: max-abs 1e-2, relative L2 2e-3."""
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


def run(env, layer, plan=None, out=None, workspace=None, expect_path=1):
    milo = env["milo"]
    pre = plan or milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max()) if layer.batch else 0
    info = milo.milo_call_info(pre.plan, layer.batch, mt)
    assert info["path"] == expect_path, info
    res = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=workspace)
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
    # exactly the threshold: 32 rows per KV head (G = 8, batch 4)
    "rows32-d128": (16, 2, 128, [512, 300, 64], (16, 64, 128), 4, [5, 64, 0, 130], True),
    # 129 rows: a second tile holding one row
    "rows129-d128": (3, 1, 128, [200, 512], (8, 40, 96, 128), 43, list(range(0, 86, 2)), True),
    # head dimension 64, ragged blocks, ranks 1 .. 64, 80 rows
    "d64-ragged": (8, 2, 64, [1, 7, 129, 64, 200], (1, 4, 7, 8, 13, 64), 20,
                   [(7 * i) % 50 for i in range(20)], True),
    # G = 7 over 448 rows (four tiles, the last half full) with short blocks
    "g7-b64": (28, 4, 128, [96, 512, 33], (16, 32, 64, 96, 128), 64, [(13 * i) % 70 for i in range(64)], False),
    # G = 5, 80 rows, long tails
    "g5-b16": (40, 8, 128, [512, 512], (32, 77, 128), 16, [1024 - 50 * i for i in range(16)], True),
    # many short blocks: shares hold many segments and cross KV heads
    "many-blocks": (28, 4, 128, [96] * 40, (4, 8, 16, 24, 128), 8, [0] * 8, True),
    # head dimension 64 with 48 rows (one spread tile) and ranks up to 64
    "d64-spread": (8, 2, 64, [300, 7, 129], (4, 16, 33, 64), 12, [(11 * i) % 90 for i in range(12)], True),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_tensor_path_matches_oracle(env, name):
    hq, hkv, d, bl, ranks, batch, tails, sep = CASES[name]
    layer = env["W"].make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                                      rank_choices=ranks, batch=batch, tail_lengths=tails,
                                      seed=zlib.crc32(name.encode()) % 1000, device="cuda",
                                      separate_kv_ranks=sep)
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), name)
    pre.close()


@pytest.mark.parametrize("batch", [10, 8])
def test_tensor_path_rank0_entries(env, batch):
    """Entries of rank 0 in K and V, in K only and in V only, next to ranks 16
    and 128, over 70 (a full tile) and 56 (a spread tile) query rows per KV
    head."""
    W = env["W"]
    rk = np.array([[0, 16], [0, 128], [16, 0], [128, 0], [0, 0]], dtype=np.int32)
    rv = np.array([[0, 0], [128, 0], [0, 16], [0, 128], [16, 0]], dtype=np.int32)
    layer = W.build_layer(14, 2, 128, [40, 512, 96, 300, 33], rk, rv, batch=batch,
                          tail_lengths=[17 * i for i in range(batch)], seed=13, device="cuda")
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), "tensor rank0")
    pre.close()


@pytest.mark.parametrize("batch", [10, 8])
def test_tensor_path_peaked_softmax(env, batch):
    """q scaled by 30: scores spread over tens of log2 units, so the rows'
    reference maxima move and V~ and O are rescaled in tensor memory (full
    and spread tiles)."""
    layer = env["W"].make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128,
                                      block_lens=[512, 77, 512, 300], rank_choices=(16, 64, 128),
                                      batch=batch, tail_lengths=[40 * i for i in range(batch)], seed=3,
                                      device="cuda", q_scale=30.0)
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), "tensor peaked")
    pre.close()


@pytest.mark.parametrize("batch", [8, 10, 20])
def test_tensor_path_outlier_records(env, batch):
    """Prefix tokens 300-309 of block 0 get scores 256 times larger, far above
    the reference each row took from its first tile: the runs holding them
    end as listed records, merged by the finish grid.  A second call on the
    same plan checks that the accumulators and lists were cleared."""
    W = env["W"]
    tails = [70 + 13 * i for i in range(batch)]
    layer = W.build_layer(14, 2, 128, [1024, 512], [[16, 16], [64, 32]], batch=batch, tail_lengths=tails,
                          seed=40 + batch, device="cuda")
    A = layer.arena
    for e in range(2):
        r = int(layer.rank_k[e])
        off = int(layer.off_ck[e])
        A[off + 300 * r:off + 310 * r] *= 256.0
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), ref, "tensor outlier")
    out2, _ = run(env, layer, plan=pre)
    compare(out2.cpu().numpy(), ref, "tensor outlier again")
    pre.close()


def test_tensor_path_repeated_and_graph_captured(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128,
                               block_lens=[512, 256, 99], rank_choices=(16, 64, 128),
                               batch=12, tail_lengths=[(31 * i) % 140 for i in range(12)], seed=8, device="cuda")
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    pre = milo.Prefix.from_layer(layer, max_batch=12)
    first, _ = run(env, layer, plan=pre)
    compare(first.cpu().numpy(), ref, "tensor repeat")
    rep_tol = 2e-5 * first.abs().max().item()
    for _ in range(3):
        again, _ = run(env, layer, plan=pre)
        assert (again - first).abs().max().item() <= rep_tol
    mt = int(np.diff(layer.tail_offsets).max())
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    out = torch.empty_like(first)
    ws = torch.empty(pre.workspace_size(12, mt), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=ws, stream=s)
        s.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            for _ in range(3):
                pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=ws, stream=s)
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert (out - first).abs().max().item() <= rep_tol
    assert pre.status() == 0
    pre.close()


@pytest.mark.parametrize("shape", [
    # (hq, hkv, d, block_lens, rank_choices, batch, tails)
    (28, 4, 128, [512, 300, 7], (0, 16, 64, 128), 1, [256]),    # 7 rows: the chunk grid by default
    (8, 8, 64, [129, 64], (1, 33, 64), 1, [5]),                  # 1 row per KV head (G = 1)
    (24, 2, 64, [200, 65], (8, 40, 64), 2, [70, 0]),             # G = 12: 24 rows, 8-row tail items
    (28, 4, 128, [128, 64], (16, 128), 64, [33] * 64),           # 448 rows: the tensor-core grid by default
])
def test_forced_paths_match_oracle_and_each_other(env, shape):
    """The same call on both paths (milo_prefix_set_tensor_min_rows): the
    chunk grid and the tensor-core grid each match the oracle, and each
    other, whatever the row count."""
    milo, W = env["milo"], env["W"]
    hq, hkv, d, bl, ranks, batch, tails = shape
    layer = W.make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl, rank_choices=ranks,
                               batch=batch, tail_lengths=tails, seed=zlib.crc32(repr(shape).encode()) % 1000,
                               device="cuda", separate_kv_ranks=True)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max())
    outs = {}
    for path, rows in ((0, 1 << 30), (1, 1)):
        pre.set_tensor_min_rows(rows)
        assert milo.milo_call_info(pre.plan, batch, mt)["path"] == path
        outs[path] = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt).cpu().numpy()
        torch.cuda.synchronize()
        assert pre.status(clear=True) == 0
        compare(outs[path], ref, f"{shape} path {path}")
    np.testing.assert_allclose(outs[0], outs[1], rtol=0, atol=1e-4)
    pre.close()


def test_call_paths(env):
    """The path milo_call_info reports for each row count of one plan."""
    milo, W = env["milo"], env["W"]
    thr = milo.milo_tensor_min_rows()
    layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128, block_lens=[64],
                               rank_choices=(16,), batch=64, tail_lengths=[0] * 64, seed=2, device="cuda")
    pre = milo.Prefix.from_layer(layer, max_batch=64)
    for batch in (1, 4, 5, 18, 19, 64):
        info = milo.milo_call_info(pre.plan, batch, 100)
        rows = batch * 7
        assert info["path"] == (1 if rows >= thr else 0), (batch, info)
        if info["path"] == 1:
            assert info["row_tiles"] == (rows + 127) // 128
            assert info["kernels"] == 3
    assert milo.milo_call_info(pre.plan, 64, 0)["kernels"] == 2
    pre.close()
