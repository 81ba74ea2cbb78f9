"""milo_attn_decode_static (the decode call that takes no workspace) against
milo_attn_decode, through the C ABI, on two calls in a row.

Tolerances as in the parity tests: max-abs 1e-2 and relative L2 2e-3."""
import zlib

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

ATOL = 1e-2
RTOL_L2 = 2e-3


@pytest.fixture(scope="module")
def env():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_29913_gb300 import build, milo, workloads
    build.build()
    milo.lib()
    return dict(milo=milo, W=workloads)


def close_enough(got, ref, what):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = np.abs(got - ref).max()
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    assert err <= ATOL and rel <= RTOL_L2, f"{what}: max-abs {err:.3e} rel-L2 {rel:.3e}"


def call_static(milo, pre, layer, toff, max_tail, out):
    rows = int(layer.tail_k.shape[0]) if max_tail > 0 else 0
    milo.milo_attn_decode_static(pre.plan, layer.q.data_ptr(), layer.batch,
                                 layer.tail_k.data_ptr() if rows else 0,
                                 layer.tail_v.data_ptr() if rows else 0,
                                 toff.data_ptr() if rows else 0, rows, max_tail if rows else 0,
                                 0.0, out.data_ptr())


@pytest.mark.parametrize("shape", [
    # (hq, hkv, d, block_lens, rank_choices, batch, tail_lengths)
    (28, 4, 128, [512, 300, 512], (16, 32, 64, 128), 2, [0, 130]),
    (14, 2, 64, [256] * 8, (8, 16, 32), 3, [5, 64, 33]),
    # 32 query rows per KV head: the prefix on the tensor-core grid, whose run
    # records sit in the built-in scratch
    (16, 2, 128, [512, 300], (16, 64, 128), 4, [5, 64, 0, 130]),
    # 20 query heads per KV head: three row groups per query on the chunk
    # grid, whose records and lists also sit in the built-in scratch
    (40, 2, 128, [200, 64, 130], (16, 64, 128), 1, [70]),
])
def test_static_scratch_matches_workspace_call(env, shape):
    milo, W = env["milo"], env["W"]
    hq, hkv, d, bl, ranks, batch, tails = shape
    layer = W.make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                               rank_choices=ranks, batch=batch, tail_lengths=tails,
                               seed=zlib.crc32(repr(shape).encode()) % 1000, device="cuda",
                               separate_kv_ranks=True)
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    max_tail = int(np.diff(layer.tail_offsets).max())
    ref = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, max_tail).cpu().numpy()
    for call in range(2):
        out = torch.full((batch, hq, d), float("nan"), device="cuda", dtype=torch.float32)
        call_static(milo, pre, layer, toff, max_tail, out)
        torch.cuda.synchronize()
        assert pre.status(clear=True) == 0, "device status word set"
        close_enough(out.cpu().numpy(), ref, f"static scratch, call {call}")
    pre.close()


def test_static_scratch_rejects_oversized_call(env):
    """A call needing more scratch than the built-in array is refused on the
    host with MILO_ERR_WORKSPACE and launches nothing (the output stays)."""
    milo, W = env["milo"], env["W"]
    batch, tail = 4, 8192   # 28 rows per KV head (the chunk grid): 128 tail items per (query, KV head)
    layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128, block_lens=[64],
                               rank_choices=(16,), batch=batch, tail_lengths=[tail] * batch,
                               seed=11, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    assert pre.workspace_size(batch, tail) > 8 << 20
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    out = torch.full((batch, 28, 128), 7.0, device="cuda", dtype=torch.float32)
    with pytest.raises(milo.MiloError) as ei:
        call_static(milo, pre, layer, toff, tail, out)
    assert ei.value.status == 8
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())
    pre.close()
