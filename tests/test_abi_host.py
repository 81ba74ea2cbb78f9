"""CPU tests of the C ABI: the library loads without a GPU, exports every
symbol the header declares, validates tables, computes the packed layout and
the static work partition -- all host logic, checked bit-exactly."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="session")
def milo():
    from paper_2609_29913_gb300 import build, milo
    build.build()
    milo.lib()
    return milo


def declared_functions():
    text = open(os.path.join(ROOT, "include", "milo.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(milo_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(milo):
    names = declared_functions()
    assert len(names) >= 10
    lib = ctypes.CDLL(milo.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(milo.EXPORTS) == names


def test_status_strings_and_version(milo):
    L = milo.lib()
    assert L.milo_version() >= 100
    for s in range(9):
        assert L.milo_status_string(s)
    assert L.milo_status_string(0) == b"ok"


def table(block_len, rk, rv=None, hkv=1, d=64, gap=0, base=0, arena_elems=None):
    """Logical row-major layout with optional gaps (multiples of 8)."""
    block_len = list(block_len)
    rk = np.asarray(rk).reshape(-1)
    rv = rk if rv is None else np.asarray(rv).reshape(-1)
    offs = np.zeros((len(rk), 4), np.int64)
    cur = base
    for b, n in enumerate(block_len):
        for g in range(hkv):
            e = b * hkv + g
            for f, sz in enumerate((n * rk[e], rk[e] * d, n * rv[e], rv[e] * d)):
                offs[e, f] = cur
                cur += int(sz) + ((-int(sz)) % 8) + gap
    return dict(num_kv_heads=hkv, head_dim=d, block_len=block_len, rank_k=rk, rank_v=rv,
                off_ck=offs[:, 0], off_pk=offs[:, 1], off_cv=offs[:, 2], off_pv=offs[:, 3],
                arena_ptr=0x10000, arena_elems=cur if arena_elems is None else arena_elems)


def ht(milo, **kw):
    return milo.HostTable(**kw)


def test_validate_accepts_good_tables(milo):
    assert milo.milo_validate_table(ht(milo, **table([7, 64, 129], [1, 8, 64], [13, 0, 64]))) == 0
    assert milo.milo_validate_table(ht(milo, **table([512] * 3, [16, 32, 128] * 2, hkv=2, d=128, gap=8))) == 0
    empty = table([], [])
    assert milo.milo_validate_table(ht(milo, **empty)) == 0


@pytest.mark.parametrize("mutate,code", [
    (lambda t: t.update(rank_k=np.array([65, 8])), 2),        # rank > head_dim
    (lambda t: t.update(rank_v=np.array([-1, 8])), 2),        # negative rank
    (lambda t: t.update(block_len=[0, 9]), 2),                # empty block
    (lambda t: t.update(block_len=[70000, 9]), 2),            # block too long
    (lambda t: t["off_pk"].__setitem__(0, t["off_pk"][0] + 4), 3),  # misaligned offset
    (lambda t: t.update(arena_elems=t["arena_elems"] - 8), 2),      # region outside arena
    (lambda t: t["off_cv"].__setitem__(1, t["off_ck"][1]), 2),      # overlapping regions
    (lambda t: t.update(head_dim=96), 4),                     # unsupported head dim
    (lambda t: t.update(num_kv_heads=0), 1),                  # no heads
    (lambda t: t.update(arena_ptr=0x10004), 3),               # misaligned arena
])
def test_validate_rejects(milo, mutate, code):
    t = table([5, 9], [4, 8])
    mutate(t)
    assert milo.milo_validate_table(ht(milo, **t)) == code


def test_packed_layout_sizes_and_alignment(milo):
    rng = np.random.default_rng(0)
    bl = list(rng.integers(1, 300, size=6))
    rk = rng.integers(0, 129, size=12)
    rv = rng.integers(0, 129, size=12)
    t = ht(milo, **table(bl, rk, rv, hkv=2, d=128))
    offs, total = milo.milo_packed_layout(t)
    r8 = lambda r: (r + 7) // 8 * 8
    sizes = []
    for e in range(12):
        n8 = (bl[e // 2] + 7) // 8 * 8
        sizes += [n8 * r8(rk[e]) * 2, r8(rk[e]) * 128 * 2, n8 * r8(rv[e]) * 2, r8(rv[e]) * 128 * 2]
    flat = offs.reshape(-1)
    assert (flat % 128 == 0).all()
    assert (np.diff(flat) >= np.array(sizes[:-1])).all()           # in order, no overlap
    assert total >= flat[-1] + sizes[-1] and total % 128 == 0
    assert total - (flat[-1] + sizes[-1]) < 128


@pytest.mark.parametrize("shares", [1, 3, 7, 152, 1000])
@pytest.mark.parametrize("shape", [
    ([512] * 64, "choice", 4, 128),
    ([7, 129, 1, 64, 65, 300], "rand", 2, 64),
    ([512] * 8, "rand", 1, 128),
])
def test_partition_covers_every_token_once(milo, shares, shape):
    """The tensor-core grid's partition: every token of every entry in exactly
    one segment, cut at 32-token boundaries; one slot per (share, KV-head
    run), slots numbered in KV-head order."""
    bl, law, hkv, d = shape
    rng = np.random.default_rng(len(bl) * 7 + shares)
    nb = len(bl)
    if law == "choice":
        rk = rng.choice([16, 32, 64, 96, 128], size=nb * hkv)
    else:
        rk = rng.integers(0, d + 1, size=nb * hkv)
    rv = rng.integers(0, d + 1, size=nb * hkv)
    t = ht(milo, **table(bl, rk, rv, hkv=hkv, d=d))
    part = milo.milo_partition_prefix(t, shares)
    cover = {}
    for e, t0, t1 in zip(part["entry"], part["t0"], part["t1"]):
        assert t0 % 32 == 0 and t0 < t1 <= bl[e // hkv]
        assert (t1 % 32 == 0) or t1 == bl[e // hkv]
        for tok in range(t0, t1):
            key = (int(e), tok)
            assert key not in cover
            cover[key] = 1
    assert len(cover) == sum(bl) * hkv
    sb = part["share_begin"]
    assert sb[0] == 0 and sb[-1] == len(part["entry"]) and (np.diff(sb) >= 0).all()
    slots = part["slot"]
    heads_of_slot = {}
    for c in range(shares):
        prev = None
        for s in range(sb[c], sb[c + 1]):
            g = int(part["entry"][s]) % hkv
            heads_of_slot.setdefault(int(slots[s]), set()).add(g)
            if prev is not None and g == prev[0]:
                assert slots[s] == prev[1]
            prev = (g, int(slots[s]))
    assert all(len(v) == 1 for v in heads_of_slot.values())
    order = [next(iter(heads_of_slot[s])) for s in sorted(heads_of_slot)]
    assert order == sorted(order)
    assert part["num_slots"] == len(heads_of_slot)


@pytest.mark.parametrize("shares", [19, 152])
def test_partition_balances_cost(milo, shares):
    """Each share's cost under the header's model (per 32-token tile of t8
    tokens t8 x (64 + r16(r^k) + r16(r^v)), plus 60000 on an entry's first
    tile), recounted from the segments, is at most total / shares plus the
    largest single tile: a tile goes to the share holding its midpoint."""
    rng = np.random.default_rng(5)
    nb, hkv, d = 64, 4, 128
    rk = rng.choice([16, 32, 64, 96, 128], size=nb * hkv)
    rv = rng.choice([16, 32, 64, 96, 128], size=nb * hkv)
    bl = [512] * nb
    t = ht(milo, **table(bl, rk, rv, hkv=hkv, d=d))
    part = milo.milo_partition_prefix(t, shares)
    r16 = lambda r: (r + 15) // 16 * 16

    def tile_cost(e, t0, n):
        t8 = (min(n - t0, 32) + 7) // 8 * 8
        return t8 * (64 + r16(rk[e]) + r16(rv[e])) + (60000 if t0 == 0 else 0)

    cost = np.zeros(shares)
    sb = part["share_begin"]
    for c in range(shares):
        for s in range(sb[c], sb[c + 1]):
            e = int(part["entry"][s])
            n = bl[e // hkv]
            for t0 in range(int(part["t0"][s]), int(part["t1"][s]), 32):
                cost[c] += tile_cost(e, t0, n)
    total = sum(tile_cost(e, t0, bl[e // hkv]) for e in range(nb * hkv) for t0 in range(0, bl[e // hkv], 32))
    assert cost.sum() == total
    biggest = max(tile_cost(e, 0, 512) for e in range(nb * hkv))
    assert cost.max() <= total / shares + biggest, (cost.max(), total / shares)
    assert (cost > 0).all()


@pytest.mark.parametrize("shape", [
    ([512] * 64, "choice", 4, 128),
    ([7, 129, 1, 64, 65, 300, 1024, 2048], "rand", 2, 64),
    ([512, 33, 1000] * 3, "rand", 3, 128),
    ([50, 70, 2048, 1], "zero", 2, 64),
])
def test_chunks_cover_every_token_once_within_budget(milo, shape):
    """The chunk grid's work list (milo_chunk_prefix): KV-head-major,
    then block order; every token of every entry exactly once; ranges start
    on 32-token boundaries; each entry uses the fewest ranges whose rows fit
    the 128 KB budget (at most 1024 tokens), and its ranges are equal up to
    the last one's remainder."""
    bl, law, hkv, d = shape
    rng = np.random.default_rng(len(bl) * 11 + hkv)
    nb = len(bl)
    if law == "choice":
        rk = rng.choice([16, 32, 64, 96, 128], size=nb * hkv)
    else:
        rk = rng.integers(0, d + 1, size=nb * hkv)
    rv = rng.integers(0, d + 1, size=nb * hkv)
    if law == "zero":  # entries of rank 0 in both K and V: tokens without coefficient rows
        rk = np.zeros(nb * hkv, dtype=np.int64)
        rv = np.zeros(nb * hkv, dtype=np.int64)
    t = ht(milo, **table(bl, rk, rv, hkv=hkv, d=d))
    ch = milo.milo_chunk_prefix(t)
    r8 = lambda r: (int(r) + 7) // 8 * 8
    # expected order: KV head g, then block b, then ascending t0
    keys = [(int(e) % hkv, int(e) // hkv, int(t0)) for e, t0 in zip(ch["entry"], ch["t0"])]
    assert keys == sorted(keys)
    per_entry = {}
    for e, t0, t1 in zip(ch["entry"], ch["t0"], ch["t1"]):
        n = bl[int(e) // hkv]
        assert t0 % 32 == 0 and t0 < t1 <= n
        per_entry.setdefault(int(e), []).append((int(t0), int(t1)))
    for b in range(nb):
        for g in range(hkv):
            e = b * hkv + g
            n = bl[b]
            ranges = per_entry.get(e, [])
            if n == 0:
                assert not ranges
                continue
            # exact cover, in order
            assert ranges[0][0] == 0 and ranges[-1][1] == n
            assert all(a[1] == c[0] for a, c in zip(ranges, ranges[1:]))
            # fewest ranges within the byte budget, and equal lengths
            row = (r8(rk[e]) + r8(rv[e])) * 2
            most = max(32, min(1024, 131072 // row // 32 * 32)) if row else 32
            assert len(ranges) == -(-n // most)
            lens = [c - a for a, c in ranges]
            assert all(L == lens[0] for L in lens[:-1]) and lens[-1] <= lens[0]
            assert lens[0] <= most and lens[0] % 32 == 0 or len(lens) == 1


def test_chunk_prefix_reports_a_short_buffer(milo):
    t = ht(milo, **table([512] * 4, [128] * 4, [128] * 4, hkv=1, d=128))
    L = milo.lib()
    n = ctypes.c_int32(0)
    assert L.milo_chunk_prefix(ctypes.byref(t.c), 0, None, None, None, ctypes.byref(n)) == 0
    assert n.value == 8  # 512 tokens at ranks 128 + 128: two 256-token ranges per entry
    buf = (ctypes.c_int32 * 4)()
    assert L.milo_chunk_prefix(ctypes.byref(t.c), 4, buf, None, None, ctypes.byref(n)) == 1
    assert n.value == 8


def test_calls_without_a_plan_fail_on_the_host(milo):
    """Every per-call entry point checks its plan before touching a device:
    a null plan is MILO_ERR_INVALID_ARG, with a message, and nothing runs."""
    L = milo.lib()
    size = ctypes.c_size_t(0)
    assert L.milo_workspace_size(None, 1, 0, ctypes.byref(size)) == 1
    assert L.milo_attn_decode(None, None, 1, None, None, None, 0, 0, ctypes.c_float(0.0), None, None, 0,
                              None) == 1
    assert b"null" in L.milo_last_error_message()
    assert L.milo_attn_decode_static(None, None, 1, None, None, None, 0, 0, ctypes.c_float(0.0), None,
                                     None) == 1
    code = ctypes.c_int32(0)
    assert L.milo_get_device_status(None, None, 0, ctypes.byref(code)) == 1
    info = milo.PrefixInfoC()
    assert L.milo_prefix_get_info(None, ctypes.byref(info)) == 1


def test_encode_layout_host(milo):
    """The compression stage's arena layout (host only): regions sized for
    min(r_max, n_b, d) ranks, 8-element aligned, in entry order, disjoint;
    the error cases."""
    bl = [512, 7, 130]
    offs, n = milo.milo_encode_layout(bl, 2, 128, r_max=96)
    assert offs.shape == (6, 4)
    cur = 0
    for b, nb in enumerate(bl):
        cap = min(96, nb, 128)
        for g in range(2):
            e = b * 2 + g
            for f, size in enumerate((nb * cap, cap * 128, nb * cap, cap * 128)):
                assert offs[e, f] == cur and offs[e, f] % 8 == 0
                cur += (size + 7) // 8 * 8
    assert n == cur
    with pytest.raises(milo.MiloError):
        milo.milo_encode_layout(bl, 2, 96, r_max=8)            # head_dim
    with pytest.raises(milo.MiloError):
        milo.milo_encode_layout([0, 4], 1, 64, r_max=8)        # empty block
    with pytest.raises(milo.MiloError):
        milo.milo_encode_layout(bl, 1, 64, r_max=8, r_min=9)   # r_min > r_max


def test_int8_entry_points_check_arguments_on_the_host(milo):
    """The INT8 entry points reject bad arguments before any device work:
    null pointers and partial groups (MILO_ERR_INVALID_ARG), misaligned
    pointers (MILO_ERR_ALIGNMENT), a null plan."""
    L = milo.lib()
    a16, a8, a4 = 1 << 20, (1 << 20) + 8, (1 << 20) + 4   # never dereferenced: the checks fail first
    assert L.milo_quantize_int8(None, 128, a8, a4, None) == 1
    assert L.milo_quantize_int8(a16, 200, a8, a4, None) == 1
    assert L.milo_quantize_int8(a16, -128, a8, a4, None) == 1
    assert L.milo_quantize_int8(a16 + 8, 128, a8, a4, None) == 3
    assert L.milo_quantize_int8(a16, 128, a8 + 4, a4, None) == 3
    assert L.milo_dequantize_int8(a8, a4 + 2, 128, a16, None) == 3
    assert L.milo_dequantize_int8(a8, a4, 128, None, None) == 1
    assert L.milo_prefix_quantize_int8(None, 0) == 1
    b = ctypes.c_int64(0)
    assert L.milo_prefix_storage_bytes(None, ctypes.byref(b), None, None) == 1


def test_tensor_threshold_setter_rejects_bad_arguments(milo):
    """milo_prefix_set_tensor_min_rows: a null plan is an argument error
    (a plan needs a device, so the rest is tested on the GPU)."""
    L = milo.lib()
    assert L.milo_prefix_set_tensor_min_rows(None, 1) == 1
    assert L.milo_prefix_set_tensor_min_rows(None, 0) == 1
    assert L.milo_tensor_min_rows() == 32


def covers_exactly(entries, t0s, t1s, bl, hkv, cut):
    """Every entry's tokens [0, n) covered once by the ranges of that entry,
    in order, each starting on a multiple of `cut` (the last ends at n)."""
    by = {}
    for e, a, b in zip(entries, t0s, t1s):
        by.setdefault(int(e), []).append((int(a), int(b)))
    assert set(by) == set(range(len(bl) * hkv))
    for e, rs in by.items():
        n = bl[e // hkv]
        assert rs[0][0] == 0 and rs[-1][1] == n, (e, rs[:2], rs[-1])
        for (a0, b0), (a1, b1) in zip(rs, rs[1:]):
            assert b0 == a1 and a0 < b0
        assert all(a % cut == 0 and a < b for a, b in rs)


@pytest.mark.parametrize("seed", range(16))
def test_work_lists_of_random_tables(milo, seed):
    """Random tables (1 to 12 blocks of 1 to 2000 tokens, 1 to 4 KV heads,
    d = 64 or 128, ranks 0 to d, K and V apart): the chunk grid's list and
    the tensor-core partition for a random share count both cover every
    token of every entry exactly once, in KV-head-major order, cut at
    32-token boundaries; no share costs more than its part of the cost line
    plus one tile."""
    rng = np.random.default_rng(1000 + seed)
    nb, hkv, d = int(rng.integers(1, 13)), int(rng.integers(1, 5)), int(rng.choice([64, 128]))
    bl = [int(x) for x in rng.integers(1, 2001, size=nb)]
    rk = rng.integers(0, d + 1, size=nb * hkv)
    rv = rng.integers(0, d + 1, size=nb * hkv)
    t = ht(milo, **table(bl, rk, rv, hkv=hkv, d=d))
    ch = milo.milo_chunk_prefix(t)
    covers_exactly(ch["entry"], ch["t0"], ch["t1"], bl, hkv, 32)
    heads = np.asarray(ch["entry"]) % hkv
    assert np.all(np.diff(heads) >= 0)                      # KV-head-major
    shares = int(rng.integers(1, 200))
    part = milo.milo_partition_prefix(t, shares)
    covers_exactly(part["entry"], part["t0"], part["t1"], bl, hkv, 32)
    r16 = lambda r: (int(r) + 15) // 16 * 16
    cost = np.zeros(shares)
    sb = part["share_begin"]
    biggest = 0
    for c in range(shares):
        for s in range(sb[c], sb[c + 1]):
            e = int(part["entry"][s])
            n = bl[e // hkv]
            for a in range(int(part["t0"][s]), int(part["t1"][s]), 32):
                tc = ((min(n - a, 32) + 7) // 8 * 8) * (64 + r16(rk[e]) + r16(rv[e])) + (60000 if a == 0 else 0)
                cost[c] += tc
                biggest = max(biggest, tc)
    assert cost.max() <= cost.sum() / shares + biggest
