"""Pins for the oracle's pre-RoPE attention (Sec. 3: the prefix keys are
compressed before the rotary position embedding, so each reconstructed
prefix key is rotated to its position before it is scored).

The checks fix the rotation from outside the oracle: closed forms on two- and
four-dimensional heads (the direction of the turn, the frequency law
theta^(-2i/d) and the pairing of dimension i with i + d/2), the identity at
position 0, the invariance of attention under a common shift of every
position, the composition and norm of rotations, and a separate pure-Python
brute force on a tiny problem."""
import math

import numpy as np
import pytest


def _arena(mats):
    parts, offs, cur = [], [], 0
    for a in mats:
        a = np.asarray(a, dtype=np.float64)
        offs.append(cur)
        parts.append(a.ravel())
        pad = (-a.size) % 8
        parts.append(np.zeros(pad))
        cur += a.size + pad
    return np.concatenate(parts), offs


def one_block(ck, pk, cv, pv, q, block_pos=None):
    """A one-KV-head problem over a single block; no tails."""
    arena, offs = _arena([ck, pk, cv, pv])
    n, d = len(ck), pk.shape[1]
    return dict(num_kv_heads=1, head_dim=d, block_len=np.array([n], np.int32),
                rank_k=np.array([pk.shape[0]], np.int32), rank_v=np.array([pv.shape[0]], np.int32),
                off_ck=np.array([offs[0]]), off_pk=np.array([offs[1]]),
                off_cv=np.array([offs[2]]), off_pv=np.array([offs[3]]),
                arena=arena, q=np.asarray(q, dtype=np.float64).reshape(1, 1, d))


def random_problem(rng, *, hq, hkv, d, block_lens, rank, batch, tail_lens):
    mats = []
    for b in range(len(block_lens)):
        for g in range(hkv):
            mats += [rng.standard_normal((block_lens[b], rank)), rng.standard_normal((rank, d)),
                     rng.standard_normal((block_lens[b], rank)), rng.standard_normal((rank, d))]
    arena, offs = _arena(mats)
    offs = np.array(offs, np.int64).reshape(-1, 4)
    toff = np.concatenate([[0], np.cumsum(tail_lens)]).astype(np.int64)
    T = max(int(toff[-1]), 1)
    E = len(block_lens) * hkv
    return dict(num_kv_heads=hkv, head_dim=d, block_len=np.array(block_lens, np.int32),
                rank_k=np.full(E, rank, np.int32), rank_v=np.full(E, rank, np.int32),
                off_ck=offs[:, 0], off_pk=offs[:, 1], off_cv=offs[:, 2], off_pv=offs[:, 3],
                arena=arena, q=rng.standard_normal((batch, hq, d)),
                tail_k=rng.standard_normal((T, hkv, d)), tail_v=rng.standard_normal((T, hkv, d)),
                tail_offsets=toff)


def softmax(x):
    e = np.exp(x - x.max())
    return e / e.sum()


@pytest.mark.parametrize("q", [(0.0, 1.0), (1.0, 0.0), (0.7, -1.3)])
def test_two_dimensional_closed_form(oracle, q):
    """d = 2: one pair, frequency theta^0 = 1.  Pre-RoPE keys (1, 0) at
    positions p = 3 .. 7 become (cos p, sin p), so the weights are
    softmax(scale (q0 cos p + q1 sin p)); q = (0, 1) gives +sin p, which fixes
    the direction of the turn."""
    n = 5
    ck = np.ones((n, 1))
    pk = np.array([[1.0, 0.0]])
    prob = one_block(ck, pk, ck, pk, q)
    _, w = oracle.attention(**prob, rope_theta=10000.0, block_pos=[3], weights=True)
    p = 3 + np.arange(n)
    scale = 1 / math.sqrt(2)
    want = softmax(scale * (q[0] * np.cos(p) + q[1] * np.sin(p)))
    np.testing.assert_allclose(w[0, 0], want, rtol=0, atol=1e-15)


@pytest.mark.parametrize("key,qdir,fn,freq", [
    (1, 3, np.sin, 0.25),   # pair (1, 3) turns at 16^(-2/4) = 1/4
    (1, 1, np.cos, 0.25),
    (0, 2, np.sin, 1.0),    # pair (0, 2) turns at 16^0 = 1
    (0, 0, np.cos, 1.0),
])
def test_four_dimensional_frequencies_and_pairing(oracle, key, qdir, fn, freq):
    """d = 4, theta = 16: dimension i pairs with i + 2 and turns at
    16^(-2i/4).  A key along e_key scored by q = e_qdir gives fn(freq p)."""
    n = 9
    ck = np.ones((n, 1))
    pk = np.zeros((1, 4))
    pk[0, key] = 1.0
    q = np.zeros(4)
    q[qdir] = 1.0
    prob = one_block(ck, pk, ck, pk, q)
    _, w = oracle.attention(**prob, rope_theta=16.0, block_pos=[11], weights=True)
    p = 11 + np.arange(n)
    want = softmax(0.5 * fn(freq * p))
    np.testing.assert_allclose(w[0, 0], want, rtol=0, atol=1e-15)


def test_position_zero_is_the_identity(oracle):
    """Blocks of one token, every block at position 0: no key turns, so the
    output equals the attention without RoPE, bit for bit."""
    rng = np.random.default_rng(5)
    prob = random_problem(rng, hq=4, hkv=2, d=8, block_lens=[1, 1, 1], rank=3, batch=2, tail_lens=[2, 0])
    plain = oracle.attention(**prob)
    rot = oracle.attention(**prob, rope_theta=500.0, block_pos=[0, 0, 0])
    assert np.array_equal(plain, rot)


def test_default_positions_are_the_concatenated_prefix(oracle):
    rng = np.random.default_rng(6)
    bl = [5, 3, 7]
    prob = random_problem(rng, hq=2, hkv=1, d=6, block_lens=bl, rank=2, batch=2, tail_lens=[1, 4])
    a = oracle.attention(**prob, rope_theta=100.0)
    b = oracle.attention(**prob, rope_theta=100.0, block_pos=[0, 5, 8])
    assert np.array_equal(a, b)
    c = oracle.attention(**prob, rope_theta=100.0, block_pos=[0, 6, 8])
    assert not np.allclose(a, c)


@pytest.mark.parametrize("shift", [1, 37, 100000])
def test_common_shift_of_every_position_leaves_attention_unchanged(oracle, shift):
    """Scores depend on positions only through their differences: moving
    every prefix block by `shift` and turning q and the tail keys by the same
    angle leaves the output unchanged (to rounding)."""
    rng = np.random.default_rng(7 + shift)
    bl = [4, 9, 6]
    prob = random_problem(rng, hq=6, hkv=2, d=8, block_lens=bl, rank=3, batch=2, tail_lens=[3, 5])
    pos = np.array([0, 50, 200])
    base = oracle.attention(**prob, rope_theta=1000.0, block_pos=pos)
    moved = dict(prob)
    moved["q"] = oracle.rope_rotate(prob["q"].reshape(-1, 8), np.full(12, shift), 1000.0).reshape(2, 6, 8)
    moved["tail_k"] = oracle.rope_rotate(prob["tail_k"].reshape(-1, 8),
                                         np.full(prob["tail_k"].shape[0] * 2, shift), 1000.0).reshape(-1, 2, 8)
    got = oracle.attention(**moved, rope_theta=1000.0, block_pos=pos + shift)
    np.testing.assert_allclose(got, base, rtol=0, atol=1e-11)
    # and the shift matters when only the keys move
    other = oracle.attention(**prob, rope_theta=1000.0, block_pos=pos + shift)
    assert np.abs(other - base).max() > 1e-6


def test_rotation_composes_and_keeps_norms(oracle):
    rng = np.random.default_rng(8)
    X = rng.standard_normal((20, 16))
    p1 = rng.integers(0, 5000, 20)
    p2 = rng.integers(0, 5000, 20)
    Y = oracle.rope_rotate(X, p1, 10000.0)
    np.testing.assert_allclose(np.linalg.norm(Y, axis=1), np.linalg.norm(X, axis=1), rtol=1e-14)
    Z = oracle.rope_rotate(Y, p2, 10000.0)
    np.testing.assert_allclose(Z, oracle.rope_rotate(X, p1 + p2, 10000.0), rtol=0, atol=1e-11)
    # inner products of two rows depend on the difference of their positions
    a, b = X[0], X[1]
    ya = oracle.rope_rotate(a[None], [123], 10000.0)[0]
    yb = oracle.rope_rotate(b[None], [100], 10000.0)[0]
    za = oracle.rope_rotate(a[None], [1023], 10000.0)[0]
    zb = oracle.rope_rotate(b[None], [1000], 10000.0)[0]
    assert abs(ya @ yb - za @ zb) < 1e-12


def brute_force_rope(prob, theta, block_pos):
    """Independent restatement with plain loops: reconstruct, turn each key
    pair by hand, softmax with math.exp."""
    d, hkv = prob["head_dim"], prob["num_kv_heads"]
    q, A = prob["q"], prob["arena"]
    batch, hq, _ = q.shape
    G = hq // hkv
    out = np.zeros_like(q)
    for i in range(batch):
        for h in range(hq):
            g = h // G
            keys, vals = [], []
            for b, n in enumerate(prob["block_len"]):
                e = b * hkv + g
                r = int(prob["rank_k"][e])
                ck = A[prob["off_ck"][e]:prob["off_ck"][e] + n * r].reshape(n, r)
                pk = A[prob["off_pk"][e]:prob["off_pk"][e] + r * d].reshape(r, d)
                cv = A[prob["off_cv"][e]:prob["off_cv"][e] + n * r].reshape(n, r)
                pv = A[prob["off_pv"][e]:prob["off_pv"][e] + r * d].reshape(r, d)
                for t in range(n):
                    k = [sum(ck[t, j] * pk[j, c] for j in range(r)) for c in range(d)]
                    rot = list(k)
                    for m in range(d // 2):
                        ang = (block_pos[b] + t) * theta ** (-2.0 * m / d)
                        rot[m] = k[m] * math.cos(ang) - k[m + d // 2] * math.sin(ang)
                        rot[m + d // 2] = k[m + d // 2] * math.cos(ang) + k[m] * math.sin(ang)
                    keys.append(rot)
                    vals.append([sum(cv[t, j] * pv[j, c] for j in range(r)) for c in range(d)])
            t0, t1 = prob["tail_offsets"][i], prob["tail_offsets"][i + 1]
            for t in range(t0, t1):
                keys.append(list(prob["tail_k"][t, g]))
                vals.append(list(prob["tail_v"][t, g]))
            s = [sum(q[i, h, c] * k[c] for c in range(d)) / math.sqrt(d) for k in keys]
            mx = max(s)
            w = [math.exp(x - mx) for x in s]
            z = sum(w)
            out[i, h] = [sum(w[t] * vals[t][c] for t in range(len(w))) / z for c in range(d)]
    return out


def test_matches_brute_force(oracle):
    rng = np.random.default_rng(9)
    prob = random_problem(rng, hq=4, hkv=2, d=6, block_lens=[3, 5, 2], rank=2, batch=2, tail_lens=[2, 3])
    pos = [10, 4, 77]
    got = oracle.attention(**prob, rope_theta=50.0, block_pos=pos)
    np.testing.assert_allclose(got, brute_force_rope(prob, 50.0, pos), rtol=0, atol=1e-12)


def test_argument_errors(oracle):
    rng = np.random.default_rng(10)
    prob = random_problem(rng, hq=2, hkv=1, d=6, block_lens=[3], rank=2, batch=1, tail_lens=[1])
    with pytest.raises(ValueError):
        oracle.attention(**prob, rope_theta=100.0, form="rankspace")
    with pytest.raises(ValueError):
        oracle.attention(**prob, rope_theta=100.0, block_pos=[0, 1])
    with pytest.raises(RuntimeError):
        oracle.attention(**prob, rope_theta=100.0, block_pos=[-1])
    odd = random_problem(rng, hq=1, hkv=1, d=5, block_lens=[2], rank=1, batch=1, tail_lens=[0])
    with pytest.raises(RuntimeError):
        oracle.attention(**odd, rope_theta=100.0)
    with pytest.raises(RuntimeError):
        oracle.rope_rotate(np.zeros((2, 4)), [0, 1], -1.0)
