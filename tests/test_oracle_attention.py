"""Pins for the oracle's attention (Eq. 1 over Alg. 1's reconstructed blocks).

Each check fixes the oracle against something other than itself: a separate
pure-Python brute force, hand-worked values, closed forms, the full-rank SVD
invariant, permutation invariance, and the equivalence of a dense tail with
an identity-basis block."""
import json
import math
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _layout(entries):
    """Pack a list of 2-D float arrays into an fp64 arena; 8-aligned offsets."""
    parts, offs, cur = [], [], 0
    for a in entries:
        a = np.asarray(a, dtype=np.float64)
        offs.append(cur)
        parts.append(a.ravel())
        pad = (-a.size) % 8
        parts.append(np.zeros(pad))
        cur += a.size + pad
    return (np.concatenate(parts) if parts else np.zeros(8)), offs


def make_problem(rng, *, hq, hkv, d, block_lens, ranks_k, ranks_v, batch,
                 tail_lens, q_scale=1.0):
    """Random fp64 problem; factors C, P generic (not orthonormal)."""
    nb = len(block_lens)
    ents, keys = [], []
    for b in range(nb):
        for g in range(hkv):
            e = b * hkv + g
            rk, rv = ranks_k[e], ranks_v[e]
            ents += [rng.standard_normal((block_lens[b], rk)),
                     rng.standard_normal((rk, d)),
                     rng.standard_normal((block_lens[b], rv)),
                     rng.standard_normal((rv, d))]
    arena, offs = _layout(ents)
    offs = np.array(offs, dtype=np.int64).reshape(-1, 4) if ents else np.zeros((0, 4), np.int64)
    toff = np.concatenate([[0], np.cumsum(tail_lens)]).astype(np.int64)
    T = int(toff[-1])
    return dict(num_kv_heads=hkv, head_dim=d,
                block_len=np.array(block_lens, np.int32),
                rank_k=np.array(ranks_k, np.int32), rank_v=np.array(ranks_v, np.int32),
                off_ck=offs[:, 0], off_pk=offs[:, 1], off_cv=offs[:, 2], off_pv=offs[:, 3],
                arena=arena, q=q_scale * rng.standard_normal((batch, hq, d)),
                tail_k=rng.standard_normal((max(T, 1), hkv, d)),
                tail_v=rng.standard_normal((max(T, 1), hkv, d)),
                tail_offsets=toff)


def brute_force(p, scale=None):
    """Independent restatement in plain Python loops: reconstruct every block
    element by element, then softmax attention with math.exp."""
    hkv, d = p["num_kv_heads"], p["head_dim"]
    q = p["q"]
    batch, hq, _ = q.shape
    G = hq // hkv
    sc = 1.0 / math.sqrt(d) if scale is None else scale
    A = p["arena"]
    out = np.zeros((batch, hq, d))
    for i in range(batch):
        for h in range(hq):
            g = h // G
            keys, vals = [], []
            for b, n in enumerate(p["block_len"]):
                e = b * hkv + g
                rk, rv = int(p["rank_k"][e]), int(p["rank_v"][e])
                for t in range(n):
                    k = [sum(A[p["off_ck"][e] + t * rk + j] * A[p["off_pk"][e] + j * d + c]
                             for j in range(rk)) for c in range(d)]
                    v = [sum(A[p["off_cv"][e] + t * rv + j] * A[p["off_pv"][e] + j * d + c]
                             for j in range(rv)) for c in range(d)]
                    keys.append(k)
                    vals.append(v)
            for t in range(p["tail_offsets"][i], p["tail_offsets"][i + 1]):
                keys.append(list(p["tail_k"][t, g]))
                vals.append(list(p["tail_v"][t, g]))
            s = [sc * sum(q[i, h, c] * k[c] for c in range(d)) for k in keys]
            m = max(s)
            w = [math.exp(x - m) for x in s]
            z = sum(w)
            for c in range(d):
                out[i, h, c] = sum(w[t] * vals[t][c] for t in range(len(w))) / z
    return out


CASES = [
    dict(hq=2, hkv=1, d=4, block_lens=[3], ranks_k=[2], ranks_v=[3], batch=1, tail_lens=[0]),
    dict(hq=4, hkv=2, d=5, block_lens=[2, 5, 1], ranks_k=[1, 2, 5, 4, 1, 1],
         ranks_v=[2, 2, 3, 5, 1, 1], batch=2, tail_lens=[3, 0]),
    dict(hq=3, hkv=1, d=8, block_lens=[9, 4], ranks_k=[8, 3], ranks_v=[7, 4], batch=1, tail_lens=[2]),
    dict(hq=2, hkv=2, d=3, block_lens=[], ranks_k=[], ranks_v=[], batch=2, tail_lens=[1, 4]),
    dict(hq=6, hkv=3, d=6, block_lens=[7, 7], ranks_k=[0, 6, 3, 2, 6, 1],
         ranks_v=[6, 0, 1, 6, 2, 3], batch=1, tail_lens=[5]),
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_dense_matches_brute_force(oracle, case):
    rng = np.random.default_rng(100 + case)
    p = make_problem(rng, **CASES[case])
    ref = brute_force(p)
    got = oracle.attention(**p)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("case", range(len(CASES)))
def test_rankspace_matches_dense(oracle, case):
    rng = np.random.default_rng(200 + case)
    p = make_problem(rng, **CASES[case])
    a = oracle.attention(**p, form="dense")
    b = oracle.attention(**p, form="rankspace")
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


def test_hand_worked_example(oracle):
    gold = json.load(open(os.path.join(GOLDEN, "attention_hand_example.json")))
    arena, offs = _layout([gold["C_K"], gold["P_K"], gold["C_V"], gold["P_V"]])
    q = np.array([[[math.sqrt(2.0) * math.log(3.0), 0.0]]])
    base = dict(num_kv_heads=1, head_dim=2, block_len=np.array(gold["block_len"]),
                rank_k=np.array(gold["rank"]), rank_v=np.array(gold["rank"]),
                off_ck=[offs[0]], off_pk=[offs[1]], off_cv=[offs[2]], off_pv=[offs[3]],
                arena=arena, q=q)
    out = oracle.attention(**base)
    np.testing.assert_allclose(out[0, 0], gold["expected_no_tail"], atol=1e-14)
    out, w = oracle.attention(**base, tail_k=np.array(gold["tail_k"])[:, None, :],
                              tail_v=np.array(gold["tail_v"])[:, None, :],
                              tail_offsets=np.array([0, 1]), weights=True)
    np.testing.assert_allclose(out[0, 0], gold["expected_with_tail"], atol=1e-14)
    np.testing.assert_allclose(w[0, 0], gold["expected_weights_with_tail"], atol=1e-15)


def test_zero_query_gives_mean_value(oracle):
    """q = 0: all scores equal, so out = mean of all value rows; per block the
    mean of V^ = (mean of C^V rows) P^V."""
    rng = np.random.default_rng(7)
    p = make_problem(rng, **CASES[1])
    p["q"] = np.zeros_like(p["q"])
    out = oracle.attention(**p)
    d, hkv = p["head_dim"], p["num_kv_heads"]
    G = p["q"].shape[1] // hkv
    A = p["arena"]
    for i in range(p["q"].shape[0]):
        for g in range(hkv):
            total, count = np.zeros(d), 0
            for b, n in enumerate(p["block_len"]):
                e = b * hkv + g
                rv = p["rank_v"][e]
                C = A[p["off_cv"][e]:p["off_cv"][e] + n * rv].reshape(n, rv)
                P = A[p["off_pv"][e]:p["off_pv"][e] + rv * d].reshape(rv, d)
                total += n * (C.mean(axis=0) @ P)
                count += n
            t0, t1 = p["tail_offsets"][i], p["tail_offsets"][i + 1]
            total += p["tail_v"][t0:t1, g].sum(axis=0)
            count += t1 - t0
            for hh in range(G):
                np.testing.assert_allclose(out[i, g * G + hh], total / count, rtol=1e-12, atol=1e-13)


def test_single_token_returns_its_value(oracle):
    rng = np.random.default_rng(8)
    p = make_problem(rng, hq=3, hkv=1, d=6, block_lens=[1], ranks_k=[4], ranks_v=[5],
                     batch=1, tail_lens=[0])
    out = oracle.attention(**p)
    A = p["arena"]
    v = A[p["off_cv"][0]:p["off_cv"][0] + 5] @ A[p["off_pv"][0]:p["off_pv"][0] + 30].reshape(5, 6)
    for h in range(3):
        np.testing.assert_allclose(out[0, h], v, rtol=1e-13, atol=1e-14)


def test_weights_row_stochastic_and_reproduce_output(oracle):
    rng = np.random.default_rng(9)
    p = make_problem(rng, **CASES[2], q_scale=3.0)
    out, w = oracle.attention(**p, weights=True)
    assert (w >= 0).all()
    np.testing.assert_allclose(w.sum(axis=-1), 1.0, atol=1e-15)
    # out = sum_t w_t v_t with v_t from an explicit dense value list
    d = p["head_dim"]
    A = p["arena"]
    vals = []
    for b, n in enumerate(p["block_len"]):
        rv = p["rank_v"][b]
        C = A[p["off_cv"][b]:p["off_cv"][b] + n * rv].reshape(n, rv)
        P = A[p["off_pv"][b]:p["off_pv"][b] + rv * d].reshape(rv, d)
        vals.append(C @ P)
    vals.append(p["tail_v"][0:2, 0])
    V = np.concatenate(vals)
    np.testing.assert_allclose(out[0], w[0] @ V, rtol=1e-12, atol=1e-13)


def test_full_rank_factors_reproduce_uncompressed_attention(oracle):
    """Full-rank SVD factors (r = min(n, d)) of dense K, V blocks give the
    uncompressed attention (Eq. 1 on the original K, V) to ~1e-12."""
    rng = np.random.default_rng(10)
    d, blocks = 6, [5, 9, 6, 1]
    K = [rng.standard_normal((n, d)) for n in blocks]
    V = [rng.standard_normal((n, d)) for n in blocks]
    full = sum(min(n, d) for n in blocks)
    comp = oracle.compress_blocks(K, V, R_tot_k=full, R_tot_v=full, r_min=0, r_max=d)
    assert list(comp["rank_k"]) == [min(n, d) for n in blocks]
    q = rng.standard_normal((2, 3, d))
    out = oracle.attention(**{k: comp[k] for k in ("num_kv_heads", "head_dim", "block_len",
                                                   "rank_k", "rank_v", "off_ck", "off_pk",
                                                   "off_cv", "off_pv", "arena")}, q=q)
    Kd, Vd = np.concatenate(K), np.concatenate(V)
    s = np.einsum("ihc,tc->iht", q, Kd) / math.sqrt(d)
    w = np.exp(s - s.max(axis=-1, keepdims=True))
    ref = np.einsum("iht,tc->ihc", w, Vd) / w.sum(axis=-1)[..., None]
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_block_order_permutation_invariance(oracle):
    rng = np.random.default_rng(11)
    p = make_problem(rng, **CASES[1])
    base = oracle.attention(**p)
    nb, hkv = len(p["block_len"]), p["num_kv_heads"]
    perm = [2, 0, 1]
    q = dict(p)
    q["block_len"] = p["block_len"][perm]
    idx = np.array([b * hkv + g for b in perm for g in range(hkv)])
    for k in ("rank_k", "rank_v", "off_ck", "off_pk", "off_cv", "off_pv"):
        q[k] = np.asarray(p[k])[idx]
    np.testing.assert_allclose(oracle.attention(**q), base, rtol=1e-13, atol=1e-14)


@pytest.mark.parametrize("cut", [1, 3, 4])
def test_block_split_invariance(oracle, cut):
    """Cutting a block's tokens into two table entries that share its P^K and
    P^V (the C rows split at the cut) leaves the attention unchanged: the
    softmax of Eq. 1 does not depend on how the tokens are grouped, which is
    what the split-K decode and its log-sum-exp merge rely on."""
    rng = np.random.default_rng(12)
    p = make_problem(rng, **CASES[1])
    base = oracle.attention(**p)
    hkv = p["num_kv_heads"]
    b = 1  # the 5-token block
    n = int(p["block_len"][b])
    assert 0 < cut < n
    lens = list(p["block_len"][:b]) + [cut, n - cut] + list(p["block_len"][b + 1:])
    q = dict(p)
    q["block_len"] = np.array(lens, np.int32)
    cols = {k: [] for k in ("rank_k", "rank_v", "off_ck", "off_pk", "off_cv", "off_pv")}
    for bb in range(len(p["block_len"])):
        parts = [(0, cut), (cut, n)] if bb == b else [(0, int(p["block_len"][bb]))]
        for t0, _ in parts:
            for g in range(hkv):
                e = bb * hkv + g
                rk, rv = int(p["rank_k"][e]), int(p["rank_v"][e])
                cols["rank_k"].append(rk)
                cols["rank_v"].append(rv)
                cols["off_ck"].append(int(p["off_ck"][e]) + t0 * rk)  # C is row-major [n][r]
                cols["off_cv"].append(int(p["off_cv"][e]) + t0 * rv)
                cols["off_pk"].append(int(p["off_pk"][e]))
                cols["off_pv"].append(int(p["off_pv"][e]))
    for k, v in cols.items():
        q[k] = np.array(v, np.int32 if k.startswith("rank") else np.int64)
    np.testing.assert_allclose(oracle.attention(**q), base, rtol=1e-13, atol=1e-14)


def test_tail_equals_identity_basis_block(oracle):
    """A dense tail K, V is the same as a full-rank block with C = K, P = I."""
    rng = np.random.default_rng(12)
    d, T = 5, 4
    kt, vt = rng.standard_normal((T, 1, d)), rng.standard_normal((T, 1, d))
    q = rng.standard_normal((1, 2, d))
    arena, offs = _layout([kt[:, 0], np.eye(d), vt[:, 0], np.eye(d)])
    as_block = oracle.attention(num_kv_heads=1, head_dim=d, block_len=[T], rank_k=[d],
                                rank_v=[d], off_ck=[offs[0]], off_pk=[offs[1]],
                                off_cv=[offs[2]], off_pv=[offs[3]], arena=arena, q=q)
    as_tail = oracle.attention(num_kv_heads=1, head_dim=d, block_len=[], rank_k=[], rank_v=[],
                               off_ck=[], off_pk=[], off_cv=[], off_pv=[], arena=np.zeros(8),
                               q=q, tail_k=kt, tail_v=vt, tail_offsets=[0, T])
    np.testing.assert_allclose(as_block, as_tail, rtol=1e-14, atol=1e-15)


def test_peaked_softmax_is_stable(oracle):
    """A huge query: weights concentrate on the best-scoring key, no overflow."""
    rng = np.random.default_rng(13)
    p = make_problem(rng, **CASES[2], q_scale=1e4)
    out, w = oracle.attention(**p, weights=True)
    assert np.isfinite(out).all()
    top = w[0].argmax(axis=-1)
    assert (w[0, np.arange(w.shape[1]), top] > 0.999).all()


def test_default_scale_is_inverse_sqrt_head_dim(oracle):
    rng = np.random.default_rng(14)
    p = make_problem(rng, **CASES[0])
    np.testing.assert_array_equal(oracle.attention(**p),
                                  oracle.attention(**p, scale=1.0 / math.sqrt(p["head_dim"])))
    assert not np.allclose(oracle.attention(**p), oracle.attention(**p, scale=1.0))


def test_bf16_inputs_widen_exactly(oracle):
    """bf16 bit patterns give bit-identical results to the same values in fp64."""
    rng = np.random.default_rng(15)
    p = make_problem(rng, **CASES[1])
    to_bits = lambda a: (np.asarray(a, np.float32).view(np.uint32) >> 16).astype(np.uint16)
    from_bits = lambda b: (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    pb = dict(p)
    pf = dict(p)
    for k in ("arena", "q", "tail_k", "tail_v"):
        pb[k] = to_bits(p[k])
        pf[k] = from_bits(pb[k])
    np.testing.assert_array_equal(oracle.attention(**pb), oracle.attention(**pf))


def test_argument_errors(oracle):
    rng = np.random.default_rng(16)
    p = make_problem(rng, **CASES[0])
    bad = dict(p, rank_k=np.array([5]))      # rank > head_dim
    with pytest.raises(RuntimeError):
        oracle.attention(**bad)
    bad = dict(p, num_kv_heads=3)             # Hq not a multiple of Hkv
    with pytest.raises(RuntimeError):
        oracle.attention(**bad)
    empty = dict(p, block_len=[], rank_k=[], rank_v=[], off_ck=[], off_pk=[], off_cv=[],
                 off_pv=[], tail_offsets=np.array([0, 0]))
    with pytest.raises(RuntimeError):        # softmax over no tokens
        oracle.attention(**empty)
