"""GPU tests of the INT8 storage of the factors (Sec. 5.3, Table 2, "MILO +
INT8"), through the C ABI:

- milo_quantize_int8 on a plan's packed arena gives, bit for bit, the codes
  and group parameters of the oracle's quantiser applied to the same factors
  (8 x 8 tiles of the logical C and P matrices, zero-padded), and
  milo_dequantize_int8 gives the oracle's read-back values bit for bit;
- a plan held as INT8 in device memory decodes from its codes directly (the
  chunk grid) like the oracle's attention over the read-back factors, and
  like its staged decode;
- a plan held as INT8 (device memory, or mapped pinned host memory read over
  the chip-to-chip link) and staged decodes like the oracle's attention over
  the read-back factors (max-abs 1e-2, relative L2 2e-3: the decode bar), on
  the chunk path and the tensor-core path, eagerly and graph-captured, with
  two staging buffers overlapped with decode;
- bytes at rest, and argument errors."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import milo_int8 as Q  # noqa: E402

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


def compare(got, ref, what=""):
    got = np.asarray(got, dtype=np.float64)
    assert np.isfinite(got).all(), what
    err = np.abs(got - ref).max()
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    assert err <= ATOL and rel <= RTOL_L2, f"{what}: max-abs {err:.3e} rel-L2 {rel:.3e}"


def arena_view(pre):
    info = pre.info
    total = int(info["packed_bytes"])

    class _View:
        __cuda_array_interface__ = dict(shape=(total,), typestr="|u1", data=(info["packed_arena"], False), version=3)
    return torch.as_tensor(_View(), device="cuda")


def packed_form(arena_bits, offs, total, table):
    """A logical arena (bf16 bits) in the packed layout of milo_packed_layout:
    8x8 tiles, row-major over [token or rank group][rank or column group],
    zero padding."""
    out = np.zeros(total // 2, dtype=np.uint16)
    for e, facs in enumerate(Q.factor_shapes(**table)):
        for f, (loff, rows, cols) in enumerate(facs):
            if rows * cols == 0:
                continue
            T = Q.tiles(arena_bits[loff:loff + rows * cols], rows, cols)
            base = int(offs[e, f]) // 2
            out[base:base + T.size] = T.reshape(-1)
    return out


def oracle_reference(env, layer):
    """The oracle's attention over the factors read back from INT8."""
    bits = layer.to_numpy_bits()
    deq, _ = Q.quantize_arena(arena=bits["arena"], **layer.table_arrays())
    bits["arena"] = deq
    return env["oracle"].attention(**bits)


CASES = {
    # name: (hq, hkv, d, block_lens, rank_choices, batch, tails)
    "chunk-d128": (28, 4, 128, [512, 300, 64, 7], (0, 13, 64, 128), 2, [37, 0]),
    "chunk-d64": (8, 2, 64, [129, 1, 65], (1, 7, 8, 64), 1, [5]),
    "tensor-d128": (28, 4, 128, [512, 256, 99], (16, 64, 128), 12, [(13 * i) % 70 for i in range(12)]),
}


def make(env, name, seed=0):
    hq, hkv, d, bl, ranks, batch, tails = CASES[name]
    return env["W"].make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                                     rank_choices=ranks, batch=batch, tail_lengths=tails, seed=seed + 17,
                                     device="cuda")


@pytest.mark.parametrize("name", ["chunk-d128", "chunk-d64"])
def test_codes_and_read_back_match_oracle_bit_exact(env, name):
    milo = env["milo"]
    layer = make(env, name)
    table = milo.HostTable.from_layer(layer)
    pre = milo.Prefix(table, layer.num_q_heads, layer.batch)
    offs, total = milo.milo_packed_layout(table)
    packed = arena_view(pre)
    codes = torch.full((total // 2,), 0xAB, dtype=torch.uint8, device="cuda")
    params = torch.full((total // 32,), 0xCD, dtype=torch.uint8, device="cuda")
    milo.milo_quantize_int8(packed, codes, params)
    back = torch.full((total,), 0xEE, dtype=torch.uint8, device="cuda")
    milo.milo_dequantize_int8(codes, params, back)
    torch.cuda.synchronize()
    C = codes.cpu().numpy()
    Pw = params.cpu().numpy().view(np.uint32)
    B = back.cpu().numpy().view(np.uint16)
    bits = layer.to_numpy_bits()
    deq, groups = Q.quantize_arena(arena=bits["arena"], **layer.table_arrays())
    for e, facs in enumerate(Q.factor_shapes(**layer.table_arrays())):
        for f, (loff, rows, cols) in enumerate(facs):
            qc, qm, qs = groups[e][f]
            R, Cg = qc.shape[:2]
            base = int(offs[e, f])
            for i in range(R):
                for j in range(Cg):
                    t = i * Cg + j
                    got = C[base // 2 + 64 * t: base // 2 + 64 * t + 64].reshape(8, 8)
                    np.testing.assert_array_equal(got, qc[i, j], err_msg=f"codes e{e} f{f} tile {i},{j}")
                    w = int(Pw[base // 128 + t])
                    assert (w & 0xFFFF, w >> 16) == (int(qm[i, j]), int(qs[i, j])), (e, f, i, j)
            # read-back values of the real (unpadded) part of the factor
            if rows * cols:
                want = deq[loff:loff + rows * cols].reshape(rows, cols)
                tiles_got = B[base // 2: base // 2 + R * Cg * 64].reshape(R, Cg, 8, 8)
                full = tiles_got.transpose(0, 2, 1, 3).reshape(R * 8, Cg * 8)
                np.testing.assert_array_equal(full[:rows, :cols], want, err_msg=f"read-back e{e} f{f}")
    pre.close()


def test_special_groups(env):
    """Constant groups, signed zeros, a 2^k grid, extremes of bf16 range."""
    milo = env["milo"]
    rng = np.random.default_rng(3)
    groups = [np.full(64, 0x4049, np.uint16),                         # constant 3.14
              np.where(np.arange(64) % 3 == 0, 0x8000, 0).astype(np.uint16),   # -0 / +0
              Q.f32_to_bf16_rne(((rng.integers(0, 256, 64) - 128) * 2.0 ** -9).astype(np.float32)),
              Q.f32_to_bf16_rne((rng.standard_normal(64) * 1e30).astype(np.float32)),
              Q.f32_to_bf16_rne((rng.standard_normal(64) * 1e-30).astype(np.float32)),
              np.where(np.arange(64) == 9, 0x0001, 0).astype(np.uint16)]       # 1/s overflows
    groups += [Q.f32_to_bf16_rne((rng.standard_normal(64) * 10.0 ** rng.uniform(-5, 5)
                                  + rng.uniform(-3, 3)).astype(np.float32)) for _ in range(58)]
    arena = np.concatenate(groups)
    packed = torch.from_numpy(arena.view(np.uint8).copy()).cuda()
    n = len(groups)
    codes = torch.empty(n * 64, dtype=torch.uint8, device="cuda")
    params = torch.empty(n * 4, dtype=torch.uint8, device="cuda")
    back = torch.empty(n * 128, dtype=torch.uint8, device="cuda")
    milo.milo_quantize_int8(packed, codes, params)
    milo.milo_dequantize_int8(codes, params, back)
    torch.cuda.synchronize()
    C = codes.cpu().numpy().reshape(n, 64)
    Pw = params.cpu().numpy().view(np.uint32)
    B = back.cpu().numpy().view(np.uint16).reshape(n, 64)
    for g in range(n):
        qc, qm, qs = Q.quantize_group(groups[g])
        assert np.array_equal(C[g], qc), g
        assert (int(Pw[g]) & 0xFFFF, int(Pw[g]) >> 16) == (qm, qs), g
        assert np.array_equal(B[g], Q.dequantize_group(qc, qm, qs)), g


@pytest.mark.parametrize("to_host", [False, True])
@pytest.mark.parametrize("name", sorted(CASES))
def test_int8_plan_decodes_like_oracle(env, name, to_host):
    milo = env["milo"]
    layer = make(env, name, seed=5)
    ref = oracle_reference(env, layer)
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = max(int(np.diff(layer.tail_offsets).max()), 1)
    nbytes = int(pre.info["packed_bytes"])
    # the staged arena must be the oracle's read-back factors in the packed
    # layout, padding zero, bit for bit
    offs, total = milo.milo_packed_layout(milo.HostTable.from_layer(layer))
    deq, _ = Q.quantize_arena(arena=layer.to_numpy_bits()["arena"], **layer.table_arrays())
    want = packed_form(deq, offs, total, layer.table_arrays())
    pre.quantize_int8(to_host=to_host)
    st = pre.storage()
    assert st == {"bytes": nbytes // 2 + nbytes // 32, "int8": True, "on_host": to_host}
    assert pre.info["packed_arena"] is None
    if to_host:
        # codes over the link are read only by the staging kernel
        with pytest.raises(milo.MiloError):
            pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    else:
        # codes in device memory: the chunk grid reads them directly
        assert env["milo"].milo_call_info(pre.plan, layer.batch, mt)["path"] == 0
        direct = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
        torch.cuda.synchronize()
        assert pre.status() == 0
        compare(direct.cpu().numpy(), ref, f"{name} int8 read directly")
    buf = torch.full((nbytes + 256,), 0x7F, dtype=torch.uint8, device="cuda")
    pre.stage(buf)
    out = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    torch.cuda.synchronize()
    assert pre.status() == 0
    np.testing.assert_array_equal(buf[:nbytes].cpu().numpy().view(np.uint16), want)
    compare(out.cpu().numpy(), ref, f"{name} int8 host={to_host}")
    if not to_host:
        # the direct read gives the staged values: the same attention up to
        # the order of the fp32 reductions
        np.testing.assert_allclose(direct.cpu().numpy(), out.cpu().numpy(), rtol=1e-5, atol=1e-5)
        pre.stage(None)
        again = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
        torch.cuda.synchronize()
        assert milo.milo_prefix_get_info(pre.plan)["packed_arena"] is None and pre.status() == 0
        np.testing.assert_allclose(again.cpu().numpy(), direct.cpu().numpy(), rtol=1e-5, atol=1e-5)
    else:
        with pytest.raises(milo.MiloError):
            pre.stage(None)                 # host codes are never read directly
    pre.close()


DIRECT = {
    # name: (hq, hkv, d, block_lens, rank_choices, batch, tails)
    # ranks 100 and 128 on both sides: full 32 KB pieces of 256 cores (codes
    # left past the values are cleared), P rows past ranks 1, 13 and 100
    "d128-full-pieces": (28, 4, 128, [512, 300, 64, 7, 1024], (0, 1, 13, 64, 100, 128), 2, [37, 0]),
    # G = 12 over 36 rows (the tensor-core grid for a bf16 plan), d = 64
    "d64-g12": (24, 2, 64, [129, 1, 65, 600], (1, 7, 8, 33, 64), 3, [5, 0, 90]),
    # one query, no tail
    "d128-b1-no-tail": (7, 1, 128, [2048, 33], (16, 96), 1, [0]),
}


@pytest.mark.parametrize("name", sorted(DIRECT))
def test_int8_read_directly_matches_staged(env, name):
    """An INT8 plan in device memory decoded by the chunk grid straight from
    its codes (no staging) gives the oracle's attention over the read-back
    factors, and the staged decode's output up to the order of the fp32
    reductions; eager and graph-captured."""
    milo = env["milo"]
    hq, hkv, d, bl, ranks, batch, tails = DIRECT[name]
    layer = env["W"].make_random_case(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, block_lens=bl,
                                      rank_choices=ranks, batch=batch, tail_lengths=tails, seed=31,
                                      device="cuda", separate_kv_ranks=True)
    ref = oracle_reference(env, layer)
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max())
    pre.quantize_int8()
    direct = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    torch.cuda.synchronize()
    assert pre.status() == 0
    compare(direct.cpu().numpy(), ref, f"{name} read directly")
    nbytes = int(pre.info["packed_bytes"])
    buf = torch.full((nbytes + 256,), 0x7F, dtype=torch.uint8, device="cuda")
    pre.stage(buf)
    staged = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    torch.cuda.synchronize()
    np.testing.assert_allclose(direct.cpu().numpy(), staged.cpu().numpy(), rtol=1e-5, atol=1e-5)
    pre.stage(None)
    out = torch.full_like(direct, float("nan"))
    ws = torch.empty(pre.workspace_size(batch, mt), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt, out=out, workspace=ws, stream=s)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert pre.status() == 0
    np.testing.assert_allclose(out.cpu().numpy(), direct.cpu().numpy(), rtol=1e-5, atol=1e-5)
    pre.close()


def test_int8_host_two_buffers_overlapped_and_captured(env):
    """Three layers held as INT8 in host memory: layer l is dequantised over
    the link into buffer l % 2 on a copy stream while the decode stream runs
    layer l - 1; eager and graph-captured steps give the oracle's results."""
    milo, W = env["milo"], env["W"]
    layers, plans, refs = [], [], []
    for l in range(3):
        layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128, block_lens=[512, 256, 99],
                                   rank_choices=(16, 64, 128), batch=2, tail_lengths=[40, 7], seed=70 + l,
                                   device="cuda")
        layers.append(layer)
        refs.append(oracle_reference(env, layer))
        pre = milo.Prefix.from_layer(layer)
        pre.quantize_int8(to_host=True)
        plans.append(pre)
    nbytes = max(int(p.info["packed_bytes"]) for p in plans)
    bufs = [torch.empty(nbytes + 128, dtype=torch.uint8, device="cuda") for _ in range(2)]
    toffs = [torch.as_tensor(L.tail_offsets, device="cuda") for L in layers]
    outs = [torch.empty((2, 28, 128), dtype=torch.float32, device="cuda") for _ in layers]
    wss = [torch.empty(p.workspace_size(2, 40), dtype=torch.uint8, device="cuda") for p in plans]
    comp, copy = torch.cuda.Stream(), torch.cuda.Stream()
    staged = [torch.cuda.Event() for _ in layers]
    done = [torch.cuda.Event() for _ in layers]
    start = torch.cuda.Event()

    def step():
        start.record(comp)
        copy.wait_event(start)
        for l, (L, pre) in enumerate(zip(layers, plans)):
            if l >= 2:
                copy.wait_event(done[l - 2])
            pre.stage(bufs[l % 2], stream=copy)
            staged[l].record(copy)
            comp.wait_event(staged[l])
            pre.decode(L.q, L.tail_k, L.tail_v, toffs[l], 40, out=outs[l], workspace=wss[l], stream=comp)
            done[l].record(comp)
        comp.wait_stream(copy)

    comp.wait_stream(torch.cuda.current_stream())
    for _ in range(2):
        with torch.cuda.stream(comp):
            step()
    comp.synchronize()
    for l in range(3):
        compare(outs[l].cpu().numpy(), refs[l], f"eager layer {l}")
        outs[l].zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=comp):
        step()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    for l in range(3):
        compare(outs[l].cpu().numpy(), refs[l], f"graph layer {l}")
        assert plans[l].status() == 0
        plans[l].close()


def test_int8_argument_errors(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128, block_lens=[128, 64],
                               rank_choices=(16, 32), batch=1, tail_lengths=[5], seed=3, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    with pytest.raises(milo.MiloError):
        pre.stage(None)                     # a resident bf16 plan
    pre.offload()
    with pytest.raises(milo.MiloError):
        pre.quantize_int8()                 # offloaded bf16 plan
    with pytest.raises(milo.MiloError):
        pre.stage(None)                     # offloaded bf16 plans need a buffer
    pre.close()
    pre = milo.Prefix.from_layer(layer)
    pre.quantize_int8()
    with pytest.raises(milo.MiloError):
        pre.quantize_int8()                 # already INT8
    with pytest.raises(milo.MiloError):
        pre.offload()                       # INT8 plans are not offloaded as bf16
    nbytes = int(pre.info["packed_bytes"])
    buf = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(milo.MiloError):
        pre.stage(buf[:64])                 # too small
    with pytest.raises(milo.MiloError) as ei:
        pre.stage(buf[1:])                  # not 128-byte aligned
    assert ei.value.status == 3
    pre.stage(buf)
    pre.close()
    x = torch.zeros(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(milo.MiloError) as ei:
        milo.milo_quantize_int8(x[:200], x, x)   # 200 bytes: not whole groups
    assert ei.value.status == 1
    with pytest.raises(milo.MiloError) as ei:
        milo.milo_dequantize_int8(x[1:129], x, x[:128])   # codes not 8-byte aligned
    assert ei.value.status == 3


def test_int8_plan_on_the_reconstruct_path_with_pre_rope(env):
    """An INT8 plan in host memory with pre-RoPE factors, staged, decoded by
    reconstruct-then-attend: the oracle's pre-RoPE attention over its INT8
    read-back (and the static no-workspace call on the rank-space path of a
    second INT8 plan)."""
    milo, W, oracle = env["milo"], env["W"], env["oracle"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128, block_lens=[512, 200, 65],
                               rank_choices=(8, 32, 128), batch=3, tail_lengths=[5, 40, 0], seed=91,
                               device="cuda")
    bits = layer.to_numpy_bits()
    deq, _ = Q.quantize_arena(arena=bits["arena"], **layer.table_arrays())
    ref = oracle.attention(**dict(bits, arena=deq), rope_theta=1e6)
    pre = milo.Prefix.from_layer(layer)
    pre.quantize_int8(to_host=True)
    pre.set_rope(1e6)
    buf = torch.empty(int(pre.info["packed_bytes"]) + 128, dtype=torch.uint8, device="cuda")
    pre.stage(buf)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    out = pre.decode_reconstruct(layer.q, layer.tail_k, layer.tail_v, toff, 40)
    torch.cuda.synchronize()
    assert pre.status() == 0
    compare(out.cpu().numpy(), ref, "int8 pre-RoPE reconstruct")
    pre.close()

    ref_rs = oracle.attention(**dict(bits, arena=deq))
    pre = milo.Prefix.from_layer(layer)
    pre.quantize_int8()
    pre.stage(buf)
    out = torch.full((3, 14, 128), float("nan"), device="cuda")
    milo.milo_attn_decode_static(pre.plan, layer.q.data_ptr(), 3, layer.tail_k.data_ptr(), layer.tail_v.data_ptr(),
                                 toff.data_ptr(), int(layer.tail_k.shape[0]), 40, 0.0, out.data_ptr())
    torch.cuda.synchronize()
    assert pre.status() == 0
    compare(out.cpu().numpy(), ref_rs, "int8 static call")
    pre.close()
