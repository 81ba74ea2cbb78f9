"""GPU tests of the offloaded prefix (milo_prefix_offload / milo_prefix_stage:
the packed factors held in pinned host memory and copied to a device buffer
before the decode calls that read them).  The decode kernels are the same,
so the parity bar is the same: the oracle's attention over the same factors
(max-abs 1e-2, relative L2 2e-3).  The cases: a never-staged plan refuses to
decode; a staged plan decodes on the chunk path and on the tensor-core path;
two layers alternate two staging buffers on a copy stream while the decode
stream runs, repeated and graph-captured; argument errors."""
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


def compare(got, ref, what=""):
    got = np.asarray(got, dtype=np.float64)
    assert np.isfinite(got).all(), what
    err = np.abs(got - ref).max()
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    assert err <= ATOL and rel <= RTOL_L2, f"{what}: max-abs {err:.3e} rel-L2 {rel:.3e}"


def staging(pre):
    return torch.empty(int(pre.info["packed_bytes"]) + 128, dtype=torch.uint8, device="cuda")


@pytest.mark.parametrize("batch", [1, 10])
def test_offloaded_plan_decodes_after_staging(env, batch):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128, block_lens=[512, 300, 64],
                               rank_choices=(16, 64, 128), batch=batch,
                               tail_lengths=[(37 * i) % 100 for i in range(batch)], seed=31 + batch, device="cuda")
    ref = env["oracle"].attention(**layer.to_numpy_bits())
    pre = milo.Prefix.from_layer(layer)
    toff = torch.as_tensor(layer.tail_offsets, device="cuda")
    mt = int(np.diff(layer.tail_offsets).max())
    before = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    pre.offload()
    assert pre.info["packed_arena"] is None
    with pytest.raises(milo.MiloError) as ei:
        pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    assert ei.value.status == 1
    buf = staging(pre)
    pre.stage(buf)
    out = pre.decode(layer.q, layer.tail_k, layer.tail_v, toff, mt)
    torch.cuda.synchronize()
    assert pre.status() == 0
    compare(out.cpu().numpy(), ref, f"offloaded b{batch}")
    assert (out - before).abs().max().item() <= 2e-5 * before.abs().max().item()
    pre.close()


def test_two_layers_two_buffers_overlapped_and_captured(env):
    """Layer l's arena is staged into buffer l % 2 on a copy stream while the
    decode stream runs layer l - 1; buffer reuse waits for the decode two
    layers back.  Eager and graph-captured replays give the oracle's
    results."""
    milo, W, oracle = env["milo"], env["W"], env["oracle"]
    layers, plans, refs = [], [], []
    for l in range(3):
        layer = W.make_random_case(num_q_heads=28, num_kv_heads=4, head_dim=128, block_lens=[512, 256, 99],
                                   rank_choices=(16, 64, 128), batch=2, tail_lengths=[40, 7], seed=50 + l,
                                   device="cuda")
        layers.append(layer)
        refs.append(oracle.attention(**layer.to_numpy_bits()))
        pre = milo.Prefix.from_layer(layer)
        pre.offload()
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
    comp.synchronize()
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


def test_offload_argument_errors(env):
    milo, W = env["milo"], env["W"]
    layer = W.make_random_case(num_q_heads=14, num_kv_heads=2, head_dim=128, block_lens=[128, 64],
                               rank_choices=(16, 32), batch=1, tail_lengths=[5], seed=3, device="cuda")
    pre = milo.Prefix.from_layer(layer)
    buf = torch.empty(int(pre.info["packed_bytes"]) + 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(milo.MiloError):
        pre.stage(buf)                      # not offloaded
    pre.offload()
    with pytest.raises(milo.MiloError):
        pre.offload()                       # already offloaded
    with pytest.raises(milo.MiloError):
        pre.stage(buf[:64])                 # too small
    with pytest.raises(milo.MiloError) as ei:
        pre.stage(buf[1:])                  # not 128-byte aligned
    assert ei.value.status == 3
    pre.stage(buf)
    pre.close()
