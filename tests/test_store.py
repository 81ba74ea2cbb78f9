"""CPU tests of a compressed prefix at rest (paper_2609_29913_gb300.store):
the block table and the bf16 arena survive a save and load bit for bit, the
loaded table passes the library's validation and packs to the same layout,
and damaged files are refused."""
import numpy as np
import pytest

from paper_2609_29913_gb300 import store
from paper_2609_29913_gb300 import workloads as W


@pytest.fixture(scope="module")
def milo():
    from paper_2609_29913_gb300 import build, milo
    build.build()
    milo.lib()
    return milo


def layer():
    return W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=64, block_lens=[129, 1, 64, 300],
                              rank_choices=(0, 7, 16, 64), batch=1, tail_lengths=[5], seed=9, device="cpu",
                              separate_kv_ranks=True)


def saved(tmp_path, L):
    path = tmp_path / "prefix.npz"
    store.save_prefix(path, **L.table_arrays(), arena=L.arena)
    return path


def test_round_trip_is_bit_exact(tmp_path):
    L = layer()
    got = store.load_prefix(saved(tmp_path, L))
    want = L.table_arrays()
    assert got["num_kv_heads"] == want["num_kv_heads"] and got["head_dim"] == want["head_dim"]
    for k in ("block_len", "rank_k", "rank_v", "off_ck", "off_pk", "off_cv", "off_pv"):
        np.testing.assert_array_equal(got[k], np.asarray(want[k]), err_msg=k)
    np.testing.assert_array_equal(got["arena"], L.to_numpy_bits()["arena"])
    # numpy bit patterns save the same way as the bf16 tensor
    path2 = tmp_path / "again.npz"
    store.save_prefix(path2, **{k: v for k, v in got.items() if k != "arena"}, arena=got["arena"])
    np.testing.assert_array_equal(store.load_prefix(path2)["arena"], got["arena"])


def test_loaded_table_validates_and_packs_the_same(tmp_path, milo):
    L = layer()
    got = store.load_prefix(saved(tmp_path, L))
    arena = got.pop("arena")
    t_loaded = milo.HostTable(**got, arena_ptr=arena.ctypes.data, arena_elems=arena.size)
    t_orig = milo.HostTable(**L.table_arrays(), arena_ptr=arena.ctypes.data, arena_elems=arena.size)
    assert milo.milo_validate_table(t_loaded) == 0
    o1, n1 = milo.milo_packed_layout(t_loaded)
    o2, n2 = milo.milo_packed_layout(t_orig)
    assert n1 == n2 and np.array_equal(o1, o2)


def damaged(tmp_path, L, **change):
    fields = dict(L.table_arrays(), arena=L.to_numpy_bits()["arena"])
    fields.update(change)
    path = tmp_path / "bad.npz"
    extra = fields.pop("_raw", None)
    if extra is not None:
        np.savez(path, **extra)
    else:
        store.save_prefix(path, **fields)
    return path


def test_damaged_files_are_refused(tmp_path):
    L = layer()
    good = dict(np.load(saved(tmp_path, L)))
    cases = {
        "format": dict(good, format=np.array("milo-prefix/0")),
        "missing": {k: v for k, v in good.items() if k != "rank_v"},
        "dtype": dict(good, off_pk=good["off_pk"].astype(np.int32)),
        "arena dtype": dict(good, arena=good["arena"].astype(np.float32)),
        "lengths": dict(good, rank_k=good["rank_k"][:-1]),
    }
    for name, raw in cases.items():
        with pytest.raises(ValueError):
            store.load_prefix(damaged(tmp_path, L, _raw=raw))
    with pytest.raises(ValueError):
        store.save_prefix(tmp_path / "x.npz", **L.table_arrays(), arena=np.zeros(8, dtype=np.float32))


def test_empty_prefix_round_trip(tmp_path):
    """A table without blocks (a call that attends to tails only) saves and
    loads as empty arrays of the right types."""
    path = tmp_path / "empty.npz"
    z32, z64 = np.zeros(0, np.int32), np.zeros(0, np.int64)
    store.save_prefix(path, num_kv_heads=2, head_dim=128, block_len=z32, rank_k=z32, rank_v=z32, off_ck=z64,
                      off_pk=z64, off_cv=z64, off_pv=z64, arena=np.zeros(0, np.uint16))
    got = store.load_prefix(path)
    assert got["num_kv_heads"] == 2 and got["head_dim"] == 128
    assert got["block_len"].dtype == np.int32 and got["off_pv"].dtype == np.int64
    assert all(got[k].size == 0 for k in ("block_len", "rank_k", "off_ck", "arena"))
