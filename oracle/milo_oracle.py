"""ctypes front end for the fp64 CPU oracle in ``milo_oracle.c``.

TEST INFRASTRUCTURE ONLY.  The oracle is the plain, slow reference the CUDA
path is checked against.  Only the test suite, ``__graft_entry__.smoke()`` and
the benchmark's CPU-baseline leg import this module.  It shares no code with
the CUDA library and never imports it.

Every function takes and returns numpy arrays.  Factor arenas and activations
may be ``float64`` or ``uint16`` holding bf16 bit patterns (widened exactly).

Functions and the passage of the paper each follows:
  attention(..., form="dense")      Alg. 1 Stage 2 reconstruction + Eq. 1
  attention(..., form="rankspace")  the same attention in rank space (Eq. 1 + Eq. 3)
  attention(..., rope_theta=...)    pre-RoPE factors (Sec. 3): reconstructed prefix
                                    keys rotated to their positions, then Eq. 1
  rope_rotate(X, pos, theta)        that rotation of the rows of X
  svd(X)                            Eq. 3, one-sided Jacobi SVD of one block
  spectral_information(sigma, r)    Eq. 5
  allocate_ranks(...)               Eq. 6 solved by the greedy rule of Eq. 7
  compress_blocks(...)              Alg. 1 Stage 1 (SVD -> ranks -> store)
  compression_ratio(...)            Eq. 4 (exact fraction)
  kv_cache_bytes(...)               Eq. 2
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from fractions import Fraction

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "milo_oracle.c")
_LIB = os.path.join(_HERE, "libmilo_oracle.so")
_lib = None

MO_F64, MO_BF16 = 0, 1
_ERRORS = {1: "invalid argument", 2: "out of memory", 3: "infeasible budget",
           4: "Jacobi SVD did not converge"}


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp64, OpenMP) if missing or stale."""
    stale = (not os.path.exists(_LIB)
             or os.path.getmtime(_LIB) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared",
                               "-std=c11", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32, i64, dbl = ctypes.c_int, ctypes.c_int64, ctypes.c_double
        L.mo_attention_dense.argtypes = [i32] * 6 + [P] * 7 + [P] * 4 + [P, dbl, P, P, i64]
        L.mo_attention_dense.restype = i32
        L.mo_attention_dense_rope.argtypes = [i32] * 6 + [P] * 7 + [P] * 4 + [P, dbl, dbl, P, P, P, i64]
        L.mo_attention_dense_rope.restype = i32
        L.mo_rope_rotate.argtypes = [i32, i32, P, P, dbl]
        L.mo_rope_rotate.restype = i32
        L.mo_attention_rankspace.argtypes = [i32] * 6 + [P] * 7 + [P] * 4 + [P, dbl, P]
        L.mo_attention_rankspace.restype = i32
        L.mo_svd_jacobi.argtypes = [i32, i32, P, P, P, P, P]
        L.mo_svd_jacobi.restype = i32
        L.mo_spectral_information.argtypes = [i32, P, dbl]
        L.mo_spectral_information.restype = dbl
        L.mo_allocate_ranks.argtypes = [i32, P, P, i32, i32, i32, i64, dbl, i32, P]
        L.mo_allocate_ranks.restype = i32
        L.mo_compression_ratio.argtypes = [i32, P, P, P, i32, P, P]
        L.mo_compression_ratio.restype = i32
        L.mo_kv_cache_bytes.argtypes = [i64, i64, i64, i64]
        L.mo_kv_cache_bytes.restype = i64
        L.mo_max_threads.restype = i32
        L.mo_set_threads.argtypes = [i32]
        _lib = L
    return _lib


def _check(rc: int, what: str):
    if rc != 0:
        raise RuntimeError(f"oracle {what}: {_ERRORS.get(rc, rc)}")


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float64:
        return MO_F64
    if a.dtype == np.uint16:
        return MO_BF16
    raise TypeError(f"oracle inputs must be float64 or uint16 (bf16 bits), got {a.dtype}")


def set_threads(n: int) -> None:
    lib().mo_set_threads(int(n))


def max_threads() -> int:
    return int(lib().mo_max_threads())


def attention(*, num_kv_heads, head_dim, block_len, rank_k, rank_v, off_ck,
              off_pk, off_cv, off_pv, arena, q, tail_k=None, tail_v=None,
              tail_offsets=None, scale=None, form="dense", weights=False,
              rope_theta=None, block_pos=None):
    """Exact decode attention of queries ``q`` [batch, Hq, d] over a low-rank
    block prefix followed by each query's dense tail.

    With ``rope_theta`` the factors are those of pre-RoPE keys: every
    reconstructed prefix key is rotated to its position (block b's token t at
    ``block_pos[b] + t``; by default the block's start in the concatenated
    prefix) before the scores; q and the tails are taken as already rotated.
    Only the dense form does this (rank space cannot hold a per-position
    rotation).

    Returns fp64 ``out`` [batch, Hq, d] (and, with ``weights=True`` and the
    dense form, the normalised softmax weights [batch, Hq, N_prefix + T_max],
    zero beyond each query's valid length)."""
    q = np.ascontiguousarray(q)
    arena = np.ascontiguousarray(arena)
    dt = _dtype_code(arena)
    if _dtype_code(q) != dt:
        raise TypeError("arena and q must share a dtype")
    batch, hq, d = q.shape
    if d != head_dim:
        raise ValueError("q head_dim mismatch")
    i32 = lambda a: np.ascontiguousarray(a, dtype=np.int32)
    i64 = lambda a: np.ascontiguousarray(a, dtype=np.int64)
    blen, rk, rv = i32(block_len), i32(rank_k), i32(rank_v)
    ock, opk, ocv, opv = i64(off_ck), i64(off_pk), i64(off_cv), i64(off_pv)
    nblk = int(blen.shape[0])
    if tail_offsets is not None:
        toff = i64(tail_offsets)
        tk = np.ascontiguousarray(tail_k)
        tv = np.ascontiguousarray(tail_v)
        if _dtype_code(tk) != dt or _dtype_code(tv) != dt:
            raise TypeError("tails must share the arena dtype")
        tmax = int(np.max(np.diff(toff))) if batch else 0
    else:
        toff = tk = tv = None
        tmax = 0
    out = np.zeros((batch, hq, d), dtype=np.float64)
    sc = 0.0 if scale is None else float(scale)
    args = (dt, batch, hq, int(num_kv_heads), d, nblk, _ptr(blen), _ptr(rk),
            _ptr(rv), _ptr(ock), _ptr(opk), _ptr(ocv), _ptr(opv), _ptr(arena),
            _ptr(q), _ptr(tk), _ptr(tv), _ptr(toff), sc, _ptr(out))
    L = lib()
    if rope_theta is not None:
        if form != "dense":
            raise ValueError("pre-RoPE factors need the dense form")
        bpos = None if block_pos is None else i64(block_pos)
        if bpos is not None and bpos.shape != (nblk,):
            raise ValueError("block_pos must hold one position per block")
        wstride = int(blen.sum()) + tmax
        w = np.zeros((batch, hq, wstride), dtype=np.float64) if weights else None
        _check(L.mo_attention_dense_rope(*args[:-1], float(rope_theta), _ptr(bpos), args[-1],
                                         _ptr(w), wstride), "attention")
        return (out, w) if weights else out
    if form == "dense":
        wstride = int(blen.sum()) + tmax
        w = np.zeros((batch, hq, wstride), dtype=np.float64) if weights else None
        _check(L.mo_attention_dense(*args, _ptr(w), wstride), "attention")
        return (out, w) if weights else out
    if form == "rankspace":
        if weights:
            raise ValueError("weights are produced by the dense form only")
        _check(L.mo_attention_rankspace(*args), "attention")
        return out
    raise ValueError(form)


def rope_rotate(X, pos, theta: float) -> np.ndarray:
    """Rows of X ([n, d] or [..., n, d], fp64) rotated by the rotary position
    embedding, row t to position pos[t] (the rotation the pre-RoPE attention
    applies to reconstructed keys)."""
    X = np.array(X, dtype=np.float64, copy=True)
    d = X.shape[-1]
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    flat = np.ascontiguousarray(X.reshape(-1, d))
    n_rows = flat.shape[0]
    if pos.size == X.shape[-2] and flat.shape[0] != pos.size:
        pos = np.broadcast_to(pos, X.shape[:-1]).reshape(-1).copy()
    if pos.size != n_rows:
        raise ValueError("one position per row")
    _check(lib().mo_rope_rotate(n_rows, d, _ptr(flat), _ptr(pos), float(theta)), "rope_rotate")
    return flat.reshape(X.shape)


def svd(X: np.ndarray):
    """SVD of one block X (n x d), Eq. 3.  Returns (sigma[k], C[n,k], P[k,d])
    with k = min(n, d), sigma non-increasing, C = A Sigma, P = B^T."""
    X = np.ascontiguousarray(X, dtype=np.float64)
    n, d = X.shape
    k = min(n, d)
    sigma = np.zeros(k)
    C = np.zeros((n, k))
    P = np.zeros((k, d))
    sweeps = ctypes.c_int(0)
    _check(lib().mo_svd_jacobi(n, d, _ptr(X), _ptr(sigma), _ptr(C), _ptr(P),
                               ctypes.byref(sweeps)), "svd")
    return sigma, C, P


def spectral_information(sigma, r: int, eps: float) -> float:
    """H(r) of Eq. 5 for one block's sorted singular values."""
    s = np.ascontiguousarray(sigma, dtype=np.float64)
    if r > s.shape[0]:
        raise ValueError("r exceeds the number of singular values")
    return float(lib().mo_spectral_information(int(r), _ptr(s), float(eps)))


def allocate_ranks(sigmas, r_min: int, r_max: int, R_tot: int, eps: float,
                   stop_at_zero_gain: bool = False) -> np.ndarray:
    """Greedy allocation (Eq. 7) of R_tot rank units over blocks whose sorted
    singular values are ``sigmas`` (a list of 1-D arrays)."""
    nb = len(sigmas)
    ld = max([len(s) for s in sigmas] + [1])
    S = np.zeros((nb, ld))
    avail = np.zeros(nb, dtype=np.int32)
    for i, s in enumerate(sigmas):
        S[i, :len(s)] = s
        avail[i] = len(s)
    out = np.zeros(nb, dtype=np.int32)
    _check(lib().mo_allocate_ranks(nb, _ptr(avail), _ptr(S), ld, int(r_min),
                                   int(r_max), int(R_tot), float(eps),
                                   int(bool(stop_at_zero_gain)), _ptr(out)),
           "allocate_ranks")
    return out


def compression_ratio(block_len, rank_k, rank_v, head_dim: int) -> Fraction:
    """rho of Eq. 4 for per-block ranks of one head (exact)."""
    bl = np.ascontiguousarray(block_len, dtype=np.int32)
    rk = np.ascontiguousarray(rank_k, dtype=np.int32)
    rv = np.ascontiguousarray(rank_v, dtype=np.int32)
    num, den = ctypes.c_int64(0), ctypes.c_int64(0)
    _check(lib().mo_compression_ratio(int(bl.shape[0]), _ptr(bl), _ptr(rk),
                                      _ptr(rv), int(head_dim),
                                      ctypes.byref(num), ctypes.byref(den)),
           "compression_ratio")
    return Fraction(num.value, den.value)


def kv_cache_bytes(N: int, L: int, H: int, d: int) -> int:
    """M of Eq. 2: bytes of an fp16 dense KV cache."""
    return int(lib().mo_kv_cache_bytes(int(N), int(L), int(H), int(d)))


def compress_blocks(K_blocks, V_blocks, *, R_tot_k, R_tot_v, r_min, r_max,
                    eps=1e-6):
    """Alg. 1 Stage 1 for one KV head: per block, SVD of K_i and of V_i
    separately (Eq. 3), greedy ranks for the K group and the V group (Eq. 7),
    then store the rank-r truncations C = A[:, :r] Sigma[:r], P = B^T[:r].

    Returns a dict with an fp64 arena and a single-KV-head block table in the
    argument form of :func:`attention` (element offsets are 8-aligned)."""
    nb = len(K_blocks)
    d = K_blocks[0].shape[1]
    fk = [svd(K) for K in K_blocks]
    fv = [svd(V) for V in V_blocks]
    rk = allocate_ranks([f[0] for f in fk], r_min, r_max, R_tot_k, eps)
    rv = allocate_ranks([f[0] for f in fv], r_min, r_max, R_tot_v, eps)
    parts, offs = [], {"off_ck": [], "off_pk": [], "off_cv": [], "off_pv": []}
    cur = 0

    def put(a, key):
        nonlocal cur
        offs[key].append(cur)
        flat = np.ascontiguousarray(a).ravel()
        parts.append(flat)
        pad = (-flat.size) % 8
        if pad:
            parts.append(np.zeros(pad))
        cur += flat.size + pad

    for i in range(nb):
        put(fk[i][1][:, :rk[i]], "off_ck")
        put(fk[i][2][:rk[i], :], "off_pk")
        put(fv[i][1][:, :rv[i]], "off_cv")
        put(fv[i][2][:rv[i], :], "off_pv")
    arena = np.concatenate(parts) if parts else np.zeros(0)
    return dict(num_kv_heads=1, head_dim=d,
                block_len=np.array([K.shape[0] for K in K_blocks], dtype=np.int32),
                rank_k=rk, rank_v=rv, arena=arena,
                **{k: np.array(v, dtype=np.int64) for k, v in offs.items()},
                sigma_k=[f[0] for f in fk], sigma_v=[f[0] for f in fv])
