"""GPU parity of the compression stage (milo_encode: Alg. 1 Stage 1, the SVD
of Eq. 3, the allocation of Eq. 6 by the greedy of Eq. 7, the rank-r
factors) against the fp64 oracle, through the C ABI.

- Singular values: against the oracle's Jacobi SVD of the same block (fp32
  eigen-decomposition of X^T X with Rayleigh-quotient eigenvalues:
  |sigma^2 - sigma_ref^2| <= 2e-6 sigma_1^2).
- Ranks: an integer decided by floating point, so both sides decide in the
  same precision: the oracle's greedy, fed the GPU's singular values, must
  give exactly the GPU's ranks (ties included: an all-zero block).
- Factors: C P (bf16, from the arena) against the oracle's rank-r
  truncation of the same block (relative Frobenius error <= 1e-2), and the
  squared residual against the tail energy of Eq. 3 (Eckart-Young).
- End to end: a plan built from the encoded arena decodes like the oracle's
  attention over the same factors.
The cases cover head dimensions 64 and 128, blocks shorter than d (rank
capped by n_b), r_min = r_max, a budget that fills every cap, and separate K
and V budgets."""
import zlib

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

EPS = 1e-6


@pytest.fixture(scope="module")
def env(oracle):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_29913_gb300 import build, milo, workloads
    build.build()
    milo.lib()
    return dict(milo=milo, W=workloads, oracle=oracle)


def bits_to_f64(t):
    """bf16 tensor -> fp64 numpy (exact)."""
    u = t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


CASES = {
    # name: (hkv, d, block_lens, r_min, r_max, mean rank K, mean rank V, zero_blocks)
    "d128": (2, 128, [512, 300, 64, 130, 7], 4, 128, 48, 32, ()),
    "d64": (3, 64, [256, 65, 1, 100], 2, 48, 20, 28, ()),
    "fixed": (1, 128, [200, 64, 9], 16, 16, 1000, 1000, ()),
    "full": (2, 64, [70, 33, 128], 0, 64, None, None, ()),
    "zeros": (2, 128, [128, 96, 160], 3, 128, 40, 40, (1,)),
}


def encode_case(env, name):
    hkv, d, bl, rmin, rmax, mk, mv, zeros = CASES[name]
    W, milo = env["W"], env["milo"]
    k, v = W.make_dense_kv(bl, hkv, d, seed=zlib.crc32(name.encode()) % 1000, device="cuda", zero_blocks=zeros)
    caps = sum(min(rmax, n, d) for n in bl)
    bk = caps if mk is None else min(caps, mk * len(bl))
    bv = caps if mv is None else min(caps, mv * len(bl))
    enc = milo.encode(k, v, bl, r_min=rmin, r_max=rmax, budget_k=bk, budget_v=bv)
    torch.cuda.synchronize()
    return dict(k=k, v=v, enc=enc, hkv=hkv, d=d, bl=bl, rmin=rmin, rmax=rmax, budget=(bk, bv))


@pytest.mark.parametrize("name", sorted(CASES))
def test_encode_matches_oracle(env, name):
    c = encode_case(env, name)
    oracle, enc = env["oracle"], c["enc"]
    hkv, d, bl = c["hkv"], c["d"], c["bl"]
    sigma = enc["sigma"].cpu().numpy().astype(np.float64)
    arena = bits_to_f64(enc["arena"])
    starts = np.concatenate([[0], np.cumsum(bl)])
    for side, X_all in enumerate((c["k"], c["v"])):
        ranks = enc["rank_v" if side else "rank_k"]
        offc, offp = enc["off_cv" if side else "off_ck"], enc["off_pv" if side else "off_pk"]
        Xn = bits_to_f64(X_all)
        for g in range(hkv):
            gpu_sig = []
            for b, n in enumerate(bl):
                e = b * hkv + g
                X = Xn[starts[b]:starts[b + 1], g, :]
                s_ref, C_ref, P_ref = oracle.svd(X)
                kk = min(n, d)
                s = sigma[2 * e + side]
                assert np.all(np.diff(s) <= 0), "singular values not sorted"
                s1 = max(s_ref[0], 1e-30)
                assert np.abs(s[:kk] ** 2 - s_ref ** 2).max() <= 2e-6 * s1 ** 2 + 1e-12, (name, side, b, g)
                assert np.abs(s[kk:] ** 2).max(initial=0.0) <= 2e-6 * s1 ** 2 + 1e-12
                gpu_sig.append(s[:kk])
                # factors against the oracle's truncation of the same rank
                r = int(ranks[e])
                C = arena[offc[e]:offc[e] + n * r].reshape(n, r)
                P = arena[offp[e]:offp[e] + r * d].reshape(r, d)
                if r == 0 or s_ref[0] == 0.0:
                    continue
                Xr = C_ref[:, :r] @ P_ref[:r]
                rel = np.linalg.norm(C @ P - Xr) / max(np.linalg.norm(Xr), 1e-30)
                assert rel <= 1e-2, (name, side, b, g, r, rel)
                tail = float(np.sum(s_ref[r:] ** 2))
                resid = float(np.linalg.norm(X - C @ P) ** 2)
                assert abs(resid - tail) <= 1e-3 * float(np.sum(s_ref ** 2)) + 1e-12, (name, side, b, g, resid, tail)
            # the allocation decided in the GPU's precision
            want = oracle.allocate_ranks(gpu_sig, c["rmin"], c["rmax"], c["budget"][side], EPS)
            got = np.array([ranks[b * hkv + g] for b in range(len(bl))])
            assert np.array_equal(got, want), (name, side, g, got, want)
            assert got.sum() == min(c["budget"][side], sum(min(c["rmax"], n, d) for n in bl))


def test_encode_then_decode(env):
    """A plan over the encoded arena decodes like the oracle over the same
    factors (and both stay close to attention over the dense keys)."""
    milo, W, oracle = env["milo"], env["W"], env["oracle"]
    hkv, d, bl = 2, 128, [512, 256, 77]
    k, v = W.make_dense_kv(bl, hkv, d, seed=11, device="cuda", noise=0.05)
    enc = milo.encode(k, v, bl, r_min=8, r_max=128, budget_k=64 * len(bl), budget_v=64 * len(bl))
    torch.cuda.synchronize()
    table = milo.HostTable(**milo.table_args(enc))
    batch, hq = 3, 14
    q = torch.randn((batch, hq, d), device="cuda").to(torch.bfloat16)
    pre = milo.Prefix(table, hq, batch)
    out = pre.decode(q).cpu().numpy().astype(np.float64)
    assert pre.status() == 0
    bits = lambda t: t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    ref = oracle.attention(num_kv_heads=hkv, head_dim=d, block_len=enc["block_len"], rank_k=enc["rank_k"],
                           rank_v=enc["rank_v"], off_ck=enc["off_ck"], off_pk=enc["off_pk"], off_cv=enc["off_cv"],
                           off_pv=enc["off_pv"], arena=bits(enc["arena"]), q=bits(q))
    err = np.abs(out - ref).max()
    rel = np.linalg.norm(out - ref) / np.linalg.norm(ref)
    assert err <= 1e-2 and rel <= 2e-3, (err, rel)
    pre.close()


def test_encode_argument_errors(env):
    milo = env["milo"]
    k = torch.zeros((10, 1, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(milo.MiloError):
        milo.encode(k, k, [10], r_min=20, r_max=8, budget_k=100, budget_v=100)   # r_min > r_max
    with pytest.raises(milo.MiloError):
        milo.encode(k, k, [10], r_min=8, r_max=16, budget_k=4, budget_v=100)     # budget below the start
    k96 = torch.zeros((10, 1, 96), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(milo.MiloError):
        milo.encode(k96, k96, [10], r_min=0, r_max=8, budget_k=8, budget_v=8)     # head_dim 96
