"""Group-wise asymmetric INT8 storage of the low-rank factors (Sec. 5.3,
Table 2: "MILO + INT8", asymmetric INT8 quantisation applied on top of the
low-rank cache).

TEST INFRASTRUCTURE ONLY.  Plain numpy restatement of the quantiser the CUDA
path implements; imported by the test suite and the benchmark's checks, never
by the CUDA library, and sharing no code with it.

The paper names the scheme (asymmetric INT8, after FlexGen) but not its
group, rounding or parameter format.  The reading taken here:

* a group is one 8 x 8 tile of a factor matrix (C: 8 tokens x 8 ranks, P:
  8 ranks x 8 head-dimension columns), the matrix zero-padded to multiples of
  8, so a group has 64 values;
* per group the minimum m and a step s with s >= (max - m) / 255, both stored
  as bf16 (m is one of the group's bf16 values, so exact; s is the fp32
  quotient rounded up to bf16, so no code passes 255);
* code c = rint((x - m) * (1 / s)) clamped to [0, 255], an unsigned byte
  (c = 0 when s = 0, a constant group, or when 1 / s overflows fp32);
* the stored value read back is bf16(m + s c).

Because floating point decides the codes, they are taken in fp32 with the
same operations as the kernel (every step an IEEE fp32 operation rounded to
nearest even; s c is exact in fp32, as s has 8 significant bits and c at
most 8).  Every function works on bf16 bit patterns (uint16 arrays)."""
from __future__ import annotations

import numpy as np

TILE = 8
GROUP = TILE * TILE


def bf16_to_f32(bits) -> np.ndarray:
    """bf16 bit patterns -> float32 (exact)."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32)


def f32_to_bf16_rne(x) -> np.ndarray:
    """float32 -> bf16 bits, rounded to nearest even (finite inputs)."""
    u = np.array(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return r.astype(np.uint16)


def f32_to_bf16_up(x) -> np.ndarray:
    """non-negative float32 -> bf16 bits, rounded up (toward +infinity)."""
    u = np.array(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u >> 16) + ((u & 0xFFFF) != 0)
    return r.astype(np.uint16)


def tiles(F_bits, rows: int, cols: int) -> np.ndarray:
    """The matrix F (rows x cols, bf16 bits), zero-padded to multiples of 8 and
    cut into 8 x 8 tiles: returns [rows8/8, cols8/8, 8, 8] bits."""
    r8, c8 = -(-rows // TILE) * TILE, -(-cols // TILE) * TILE
    P = np.zeros((r8, c8), dtype=np.uint16)
    P[:rows, :cols] = np.asarray(F_bits, dtype=np.uint16).reshape(rows, cols)
    return P.reshape(r8 // TILE, TILE, c8 // TILE, TILE).transpose(0, 2, 1, 3).copy()


def quantize_groups(x_bits):
    """Groups of 64 values (bf16 bits, shape [..., 8, 8] or [..., 64]: the
    last axes hold one group) -> (codes uint8 of the same shape, m bits [...],
    s bits [...])."""
    x_bits = np.asarray(x_bits, dtype=np.uint16)
    shape = x_bits.shape
    lead = shape[:-2] if shape[-2:] == (TILE, TILE) else shape[:-1]
    x = bf16_to_f32(x_bits).reshape(lead + (GROUP,)).astype(np.float32)
    zero = np.float32(0.0)
    lo = (x.min(axis=-1) + zero).astype(np.float32)      # + 0 turns -0 into +0
    hi = (x.max(axis=-1) + zero).astype(np.float32)
    span = (hi - lo).astype(np.float32)
    s_bits = f32_to_bf16_up((span / np.float32(255.0)).astype(np.float32))
    s = bf16_to_f32(s_bits)
    m_bits = f32_to_bf16_rne(lo)                          # exact: lo is one of the bf16 values (or +0)
    with np.errstate(over="ignore", divide="ignore"):
        inv = (np.float32(1.0) / np.where(s > 0, s, np.float32(1.0))).astype(np.float32)
    inv = np.where((s > 0) & np.isfinite(inv), inv, np.float32(0.0)).astype(np.float32)
    # s = 0, or 1 / s beyond fp32: inv = 0 and every code 0
    t = (x - lo[..., None]).astype(np.float32)            # fp32 subtraction
    c = np.rint((t * inv[..., None]).astype(np.float32))  # fp32 product, nearest even
    codes = np.clip(c, 0, 255).astype(np.uint8).reshape(shape)
    return codes, m_bits, s_bits


def quantize_group(x_bits):
    """One group (64 values of bf16 bits, any shape) -> (codes uint8 of the
    same shape, m bits, s bits)."""
    x_bits = np.asarray(x_bits, dtype=np.uint16)
    codes, m, s = quantize_groups(x_bits.reshape(GROUP))
    return codes.reshape(x_bits.shape), int(m), int(s)


def dequantize_groups(codes, m_bits, s_bits) -> np.ndarray:
    """Codes of groups ([..., 8, 8] or [..., 64]) with their m and s bits
    ([...]) -> bf16 bits of m + s c (fp32: s c exact, one rounding for the
    sum; then to bf16, nearest even)."""
    codes = np.asarray(codes, dtype=np.uint8)
    shape = codes.shape
    m = bf16_to_f32(np.asarray(m_bits, dtype=np.uint16))
    s = bf16_to_f32(np.asarray(s_bits, dtype=np.uint16))
    c = codes.reshape(m.shape + (GROUP,)).astype(np.float32)
    prod = (s[..., None] * c).astype(np.float32)          # exact
    return f32_to_bf16_rne((m[..., None] + prod).astype(np.float32)).reshape(shape)


def dequantize_group(codes, m_bits: int, s_bits: int) -> np.ndarray:
    """Codes of one group -> bf16 bits of m + s c."""
    codes = np.asarray(codes, dtype=np.uint8)
    return dequantize_groups(codes.reshape(GROUP), np.uint16(m_bits), np.uint16(s_bits)).reshape(codes.shape)


def quantize_matrix(F_bits, rows: int, cols: int):
    """All tiles of one factor matrix.  Returns codes [R, Cg, 8, 8] uint8 and
    m, s bits [R, Cg] (R = rows8/8, Cg = cols8/8)."""
    return quantize_groups(tiles(F_bits, rows, cols))


def dequantize_matrix(codes, m, s, rows: int, cols: int) -> np.ndarray:
    """Inverse of quantize_matrix up to the quantisation error: bf16 bits
    [rows, cols] (the padding dropped)."""
    R, Cg = codes.shape[:2]
    T = dequantize_groups(codes, m, s)
    return T.transpose(0, 2, 1, 3).reshape(R * TILE, Cg * TILE)[:rows, :cols]


def factor_shapes(*, num_kv_heads, head_dim, block_len, rank_k, rank_v, off_ck, off_pk, off_cv, off_pv):
    """(offset, rows, cols) of every factor of a block table, entry by entry
    (entry e = block * num_kv_heads + head), in the order C^K, P^K, C^V, P^V."""
    out = []
    for e in range(len(rank_k)):
        n = int(block_len[e // num_kv_heads])
        rk, rv = int(rank_k[e]), int(rank_v[e])
        out.append([(int(off_ck[e]), n, rk), (int(off_pk[e]), rk, head_dim),
                    (int(off_cv[e]), n, rv), (int(off_pv[e]), rv, head_dim)])
    return out


def quantize_arena(*, arena, **table):
    """Every factor of a logical arena (bf16 bits, the block table's offsets)
    quantised and read back.  Returns (arena of the read-back values, same
    layout; list per entry of four (codes, m, s) triples)."""
    arena = np.asarray(arena, dtype=np.uint16)
    deq = arena.copy()
    groups = []
    for facs in factor_shapes(**table):
        g = []
        for off, rows, cols in facs:
            F = arena[off:off + rows * cols]
            codes, m, s = quantize_matrix(F, rows, cols)
            if rows * cols:
                deq[off:off + rows * cols] = dequantize_matrix(codes, m, s, rows, cols).reshape(-1)
            g.append((codes, m, s))
        groups.append(g)
    return deq, groups


def stored_bytes(rows: int, cols: int) -> tuple[int, int]:
    """Bytes of one factor held as bf16 tiles and as INT8 tiles (64 one-byte
    codes plus a bf16 m and a bf16 s per tile)."""
    ntiles = (-(-rows // TILE)) * (-(-cols // TILE))
    return ntiles * GROUP * 2, ntiles * (GROUP + 4)
