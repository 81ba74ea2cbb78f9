"""GPU test of a compressed prefix at rest: a plan built from a saved file
(paper_2609_29913_gb300.store.prefix_from_file) packs the same arena bit for
bit as the plan built from the layer in memory, and decodes like the oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


def packed_bytes(pre):
    info = pre.info
    total = int(info["packed_bytes"])

    class _View:
        __cuda_array_interface__ = dict(shape=(total,), typestr="|u1", data=(info["packed_arena"], False), version=3)
    return torch.as_tensor(_View(), device="cuda").cpu().numpy()


def test_plan_from_saved_prefix(tmp_path, oracle):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_29913_gb300 import build, milo, store
    from paper_2609_29913_gb300 import workloads as W
    build.build()
    layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128, block_lens=[512, 300, 7],
                               rank_choices=(0, 13, 64, 128), batch=3, tail_lengths=[40, 0, 129], seed=21,
                               device="cuda", separate_kv_ranks=True)
    path = tmp_path / "prefix.npz"
    store.save_prefix(path, **layer.table_arrays(), arena=layer.arena)
    pre = store.prefix_from_file(path, layer.num_q_heads, layer.batch)
    ref_plan = milo.Prefix.from_layer(layer)
    assert np.array_equal(packed_bytes(pre), packed_bytes(ref_plan))
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max())
    out = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    torch.cuda.synchronize()
    assert pre.status() == 0
    ref = oracle.attention(**layer.to_numpy_bits())
    got = out.double().cpu().numpy()
    assert np.abs(got - ref).max() <= 1e-2
    assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 2e-3
    pre.close()
    ref_plan.close()
