"""GPU parity of reconstruct-then-attend (milo_attn_decode_reconstruct, the
paper's own inference path: dense keys and values rebuilt from the factors,
then attended) and of its pre-RoPE variant, against the fp64 oracle, through
the C ABI.

The cases cover the ways the 8 warps of a block share rows (4 warps per
16-row fragment in groups of up to 32 query rows, 2 up to 64, 1 up to 128,
and more than one group), head dimensions 64 and 128, ragged blocks (1 to 600 tokens: partial tiles and several chunks),
ranks 0 (K, V or both) next to full ranks, a peaked softmax, outlier scores
that force the listed-record merge, calls without tails, rotation tables for
the default and for explicit block positions, the refusal of the rank-space
call on a pre-RoPE plan, the two paths alternating on one plan, repeated and
graph-captured calls, and layer 0 of the batch-1 and batch-64 workloads.
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


def run(env, layer, plan=None, out=None, workspace=None):
    milo = env["milo"]
    pre = plan or milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max()) if layer.batch else 0
    res = pre.decode_reconstruct(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=workspace)
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
    # 7 rows per KV head: one fragment, 4 warps split each tile's tokens
    "b1-g7-d128": (28, 4, 128, [512, 300, 64, 65, 1], (16, 32, 64, 96, 128), 1, [256], True),
    # 28 rows: two fragments, four warps each
    "b4-g7-d128": (28, 4, 128, [200, 600, 7], (8, 40, 96, 128), 4, [5, 64, 0, 130], True),
    # 70 rows: one group, a warp per fragment
    "b10-g7-d128": (14, 2, 128, [512, 129], (16, 64, 128), 10, [(37 * i) % 90 for i in range(10)], False),
    # 140 rows: two groups (128 + 12 rows)
    "b20-g7-d128": (28, 4, 128, [256, 77], (16, 64, 128), 20, [(41 * i) % 70 for i in range(20)], True),
    # head dimension 64, ragged blocks, ranks 1 .. 64, 48 rows (three fragments, two warps each)
    "d64-ragged": (8, 2, 64, [1, 7, 129, 64, 200], (1, 4, 7, 8, 13, 64), 12,
                   [(7 * i) % 50 for i in range(12)], True),
    # G = 5, 80 rows (five fragments), long tails
    "g5-b16": (40, 8, 128, [512, 256], (32, 77, 128), 16, [1024 - 50 * i for i in range(16)], True),
    # G = 1 and no tails
    "g1-notail": (4, 4, 128, [300, 64, 100], (16, 128), 3, [0, 0, 0], True),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_reconstruct_matches_oracle(env, name):
    hq, hkv, d, bl, ranks, batch, tails, sep = CASES[name]
    layer = env["W"].make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                                      rank_choices=ranks, batch=batch, tail_lengths=tails,
                                      seed=zlib.crc32(name.encode()) % 1000, device="cuda",
                                      separate_kv_ranks=sep)
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), name)
    pre.close()


def test_reconstruct_rank0_entries(env):
    """Entries of rank 0 in K and V, in K only and in V only, next to ranks
    16 and 128 (their keys or values reconstruct to zero)."""
    W = env["W"]
    rk = np.array([[0, 16], [0, 128], [16, 0], [128, 0], [0, 0]], dtype=np.int32)
    rv = np.array([[0, 0], [128, 0], [0, 16], [0, 128], [16, 0]], dtype=np.int32)
    for batch in (1, 10):
        layer = W.build_layer(14, 2, 128, [40, 512, 96, 300, 33], rk, rv, batch=batch,
                              tail_lengths=[17 * i for i in range(batch)], seed=13 + batch, device="cuda")
        out, pre = run(env, layer)
        compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), f"rank0 b{batch}")
        pre.close()


def test_reconstruct_peaked_softmax(env):
    layer = env["W"].make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128,
                                      block_lens=[512, 77, 512, 300], rank_choices=(16, 64, 128),
                                      batch=3, tail_lengths=[40, 0, 300], seed=3, device="cuda", q_scale=30.0)
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), env["oracle"].attention(**layer.to_numpy_bits()), "peaked")
    pre.close()


@pytest.mark.parametrize("batch", [1, 10])
def test_reconstruct_outlier_records(env, batch):
    """Prefix tokens 300-309 of block 0 score 256 times higher: the chunks
    holding them end far above the reference of the chunk that published it
    first (or the others end far below theirs), so records are listed and
    merged by the finish grid.  A second call checks that the accumulators
    and lists were cleared."""
    W = env["W"]
    layer = W.build_layer(14, 2, 128, [1024, 512], [[16, 16], [64, 32]], batch=batch,
                          tail_lengths=[70 + 13 * i for i in range(batch)], seed=40 + batch, device="cuda")
    A = layer.arena
    for e in range(2):
        r = int(layer.rank_k[e])
        off = int(layer.off_ck[e])
        A[off + 300 * r:off + 310 * r] *= 256.0
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    out, pre = run(env, layer)
    compare(out.cpu().numpy(), ref, "outlier")
    out2, _ = run(env, layer, plan=pre)
    compare(out2.cpu().numpy(), ref, "outlier again")
    pre.close()


@pytest.mark.parametrize("theta,positions", [(10000.0, None), (1e6, None), (500.0, "explicit")])
@pytest.mark.parametrize("batch,d", [(1, 128), (10, 128), (6, 64)])
def test_pre_rope_matches_oracle(env, theta, positions, batch, d):
    """Pre-RoPE factors: each reconstructed key turns to its position."""
    W = env["W"]
    bl = [512, 200, 65, 300]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=d, block_lens=bl,
                               rank_choices=(8, 32, 64, d), batch=batch,
                               tail_lengths=[(29 * i) % 100 for i in range(batch)],
                               seed=int(theta) % 97 + batch + d, device="cuda")
    pos = None if positions is None else np.array([70000, 5, 131072, 4000], dtype=np.int64)
    pre = env["milo"].Prefix.from_layer(layer)
    pre.set_rope(theta, pos)
    out, _ = run(env, layer, plan=pre)
    ref = env["oracle"].attention(**layer.to_numpy_bits(), rope_theta=theta, block_pos=pos)
    compare(out.cpu().numpy(), ref, f"rope theta {theta} positions {positions}")
    # and the rotation is not a no-op on these inputs
    plain = env["oracle"].attention(**layer.to_numpy_bits())
    assert np.abs(plain - ref).max() > 1e-3
    pre.close()


def test_pre_rope_plan_refuses_rank_space_and_clears(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128, block_lens=[256, 100],
                               rank_choices=(16, 64), batch=2, tail_lengths=[10, 20], seed=21, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    pre.set_rope(10000.0)
    with pytest.raises(milo.MiloError) as ei:
        pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, 20)
    assert ei.value.status == 4  # MILO_ERR_UNSUPPORTED
    with pytest.raises(milo.MiloError):
        pre.set_rope(-1.0)
    with pytest.raises(milo.MiloError):
        pre.set_rope(100.0, [0, -5])
    pre.set_rope(0.0)
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    compare(pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, 20).cpu().numpy(), ref, "rank space after clear")
    out, _ = run(env, layer, plan=pre)
    compare(out.cpu().numpy(), ref, "reconstruct after clear")
    pre.close()


def test_paths_alternate_on_one_plan_and_graph_capture(env):
    """Rank-space and reconstruct calls share the plan's per-call state:
    alternate them, then replay a captured graph of reconstruct calls."""
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128,
                               block_lens=[512, 256, 99], rank_choices=(16, 64, 128),
                               batch=12, tail_lengths=[(31 * i) % 140 for i in range(12)], seed=8, device="cuda")
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    pre = milo.Prefix.from_layer(layer, max_batch=12)
    mt = int(np.diff(layer.tail_offsets).max())
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    first, _ = run(env, layer, plan=pre)
    compare(first.cpu().numpy(), ref, "reconstruct")
    rep_tol = 2e-5 * first.abs().max().item()
    for _ in range(2):
        a = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
        b = pre.decode_reconstruct(layer.q, layer.tail_k, layer.tail_v, toff, mt)
        torch.cuda.synchronize()
        compare(a.cpu().numpy(), ref, "rank space between")
        assert (b - first).abs().max().item() <= rep_tol
    out = torch.empty_like(first)
    ws = torch.empty(pre.workspace_size(12, mt), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        pre.decode_reconstruct(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=ws, stream=s)
        s.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            for _ in range(3):
                pre.decode_reconstruct(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=ws,
                                       stream=s)
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert (out - first).abs().max().item() <= rep_tol
    assert pre.status() == 0
    pre.close()


@pytest.mark.parametrize("name", ["qwen7b-28L-32k-b1", "qwen7b-28L-32k-b64"])
def test_reconstruct_workload_layer0(env, name):
    """Layer 0 of the batch-1 and batch-64 workloads over the whole output."""
    W = env["W"]
    layer = W.make_config_layer(W.by_name(name), 0, device="cuda")
    out, pre = run(env, layer)
    got = out.cpu().numpy()
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    err, rel = compare(got, ref, f"{name} layer 0")
    print(f"{name} layer 0 reconstruct: max-abs {err:.3e} rel-L2 {rel:.3e}")
    pre.close()
