"""Seeded synthetic inputs for decode attention over a block-wise low-rank
KV prefix.

This module only draws random inputs; it contains none of the method's
arithmetic.  Both the CUDA path and the CPU oracle consume exactly the bytes
it produces (bf16 factors and activations, integer tables).

Logical prefix layout (one decoder layer, one arena):
  for every block b (table order) and KV head g, entry e = b * Hkv + g holds
    C^K_e  [n_b, r^k_e]  row-major   coefficients (Sigma folded in, Eq. 3)
    P^K_e  [r^k_e, d]    row-major   orthonormal basis rows
    C^V_e  [n_b, r^v_e]
    P^V_e  [r^v_e, d]
  each starting at an element offset that is a multiple of 8 (16 bytes).
  Gaps between factors are zero, or NaN when ``poison_gaps`` is set.

Recipe (stands in for the paper's Qwen2.5 many-shot KV caches, which need
model weights and datasets that are not available here):
  P = (Q of the reduced QR of a d x r standard Gaussian)^T, rounded to bf16
      (drawn and factorised on the host, so identical on every device);
  C[:, j] ~ N(0, 1/j) for j = 1..r (1/j is the variance), rounded to bf16;
  q, tail K, tail V ~ N(0, 1) in bf16; ``q_scale`` multiplies q (e.g. 30 for
  a peaked softmax).  Integer draws (ranks, tail lengths) use numpy's PCG64
  seeded with (seed, layer); floating-point draws use torch's generator on the
  target device seeded from (seed, layer).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import numpy as np
import torch

ALIGN = 8  # elements (16 bytes of bf16) between factor starts


@dataclass
class Config:
    """One synthetic workload shape."""
    name: str
    layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    num_blocks: int
    block_len: int
    rank_law: str          # "choice", "entropy_multinomial", "geometric"
    rank_choices: tuple = ()
    batch: int = 1
    tail_law: str = "fixed"  # "fixed" or "uniform"
    tail_len: int = 0
    tail_range: tuple = (0, 0)
    seed: int = 0
    description: str = ""

    @property
    def prefix_tokens(self) -> int:
        return self.num_blocks * self.block_len


# The five Qwen2.5-shaped workloads.  Seeds are 1000 + index.
CONFIGS = [
    Config("qwen0.5b-1L-2k", 1, 14, 2, 64, 8, 256, "choice", (8, 16, 32),
           batch=1, tail_len=0, seed=1000,
           description="1 layer, 14/2 heads, d=64, 8x256 prefix, r in {8,16,32}, batch 1, no tail"),
    Config("qwen7b-28L-32k-b1", 28, 28, 4, 128, 64, 512, "choice",
           (16, 32, 64, 96, 128), batch=1, tail_len=256, seed=1001,
           description="28 layers, 28/4 heads, d=128, 64x512 prefix, r in {16..128}, batch 1, tail 256"),
    Config("qwen7b-28L-32k-b64", 28, 28, 4, 128, 64, 512, "choice",
           (16, 32, 64, 96, 128), batch=64, tail_len=512, seed=1002,
           description="the qwen7b-28L-32k-b1 prefix shared by 64 queries, tail 512 each"),
    Config("qwen14b-48L-128k-b16", 48, 40, 8, 128, 256, 512,
           "entropy_multinomial", batch=16, tail_len=1024, seed=1003,
           description="48 layers, 40/8 heads, 256x512 prefix, r 32..128 mean 64, batch 16, tail 1024"),
    Config("qwen7b-1L-1M-b8", 1, 28, 4, 128, 2048, 512, "geometric", batch=8,
           tail_law="uniform", tail_range=(128, 4096), seed=1004,
           description="1 layer, 2048x512 prefix, geometric ranks 4..128 + 5% full rank, batch 8, tails U[128,4096]"),
]


def by_name(name: str) -> Config:
    """The workload called `name` (e.g. "qwen7b-28L-32k-b1")."""
    for cfg in CONFIGS:
        if cfg.name == name:
            return cfg
    raise KeyError(name)


def _np_rng(seed: int, layer: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([int(seed), int(layer)]))


def draw_ranks(cfg: Config, layer: int) -> np.ndarray:
    """Per-(block, KV head) ranks, shape [num_blocks, num_kv_heads] int32.
    K and V share the rank (the workloads state one rank per block)."""
    rng = _np_rng(cfg.seed, layer)
    nb, hk = cfg.num_blocks, cfg.num_kv_heads
    if cfg.rank_law == "choice":
        r = rng.choice(np.asarray(cfg.rank_choices), size=(nb, hk))
    elif cfg.rank_law == "entropy_multinomial":
        # r_b = 32 + multinomial share of 32 * nb extra units, p ~ e_b ~ U(0,1),
        # capped at 128 with the excess redrawn over uncapped blocks: mean 64.
        r = np.zeros((nb, hk), dtype=np.int64)
        for g in range(hk):
            e = rng.uniform(0.0, 1.0, size=nb)
            rg = 32 + rng.multinomial(32 * nb, e / e.sum())
            while (rg > 128).any():
                excess = int((rg - 128).clip(min=0).sum())
                rg = np.minimum(rg, 128)
                open_ = rg < 128
                w = np.where(open_, e, 0.0)
                rg = rg + rng.multinomial(excess, w / w.sum())
            r[:, g] = rg
    elif cfg.rank_law == "geometric":
        # Geom(p=0.05) on {1,2,...} clipped to [4,128]; floor(0.05 nb) seeded
        # blocks at full rank 128 for every KV head.
        r = np.clip(rng.geometric(0.05, size=(nb, hk)), 4, 128)
        full = rng.choice(nb, size=int(0.05 * nb), replace=False)
        r[full, :] = 128
    else:
        raise ValueError(cfg.rank_law)
    return np.asarray(r, dtype=np.int32)


def draw_tail_lengths(cfg: Config, layer: int) -> np.ndarray:
    if cfg.tail_law == "fixed":
        return np.full(cfg.batch, cfg.tail_len, dtype=np.int64)
    rng = _np_rng(cfg.seed + 7919, layer)
    lo, hi = cfg.tail_range
    return rng.integers(lo, hi + 1, size=cfg.batch).astype(np.int64)


@dataclass
class LayerInputs:
    """All inputs of one decode-attention call (one layer)."""
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    block_len: np.ndarray        # [nb] int32
    rank_k: np.ndarray           # [nb * Hkv] int32, entry b * Hkv + g
    rank_v: np.ndarray
    off_ck: np.ndarray           # [nb * Hkv] int64 element offsets
    off_pk: np.ndarray
    off_cv: np.ndarray
    off_pv: np.ndarray
    arena: torch.Tensor          # [arena_elems] bf16
    q: torch.Tensor              # [batch, Hq, d] bf16
    tail_k: Optional[torch.Tensor]  # [sum T, Hkv, d] bf16 or None
    tail_v: Optional[torch.Tensor]
    tail_offsets: np.ndarray     # [batch + 1] int64
    meta: dict = field(default_factory=dict)

    @property
    def batch(self) -> int:
        return int(self.q.shape[0])

    @property
    def num_blocks(self) -> int:
        return int(self.block_len.shape[0])

    def table_arrays(self) -> dict:
        return dict(num_kv_heads=self.num_kv_heads, head_dim=self.head_dim,
                    block_len=self.block_len, rank_k=self.rank_k,
                    rank_v=self.rank_v, off_ck=self.off_ck, off_pk=self.off_pk,
                    off_cv=self.off_cv, off_pv=self.off_pv)

    def to_numpy_bits(self) -> dict:
        """Host copies as uint16 bf16 bit patterns, in the oracle's argument form."""
        bits = lambda t: None if t is None else t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        d = self.table_arrays()
        d.update(arena=bits(self.arena), q=bits(self.q))
        if self.tail_k is not None and int(self.tail_offsets[-1]) > 0:
            d.update(tail_k=bits(self.tail_k), tail_v=bits(self.tail_v),
                     tail_offsets=self.tail_offsets)
        elif self.batch and self.num_blocks == 0:
            d.update(tail_k=bits(self.tail_k), tail_v=bits(self.tail_v),
                     tail_offsets=self.tail_offsets)
        return d


def _torch_gen(device, seed: int, layer: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + int(layer) * 7_919 + 12_345) % (2 ** 62))
    return g


def _orthonormal_rows(m: int, r: int, d: int, gen_cpu, device) -> torch.Tensor:
    """m independent r x d matrices with orthonormal rows (fp32), drawn and
    factorised on the host (identical on every device), then moved."""
    a = torch.randn((m, d, r), generator=gen_cpu, dtype=torch.float32)
    qm, _ = torch.linalg.qr(a, mode="reduced")    # [m, d, r]
    return qm.transpose(1, 2).contiguous().to(device)  # [m, r, d]


def build_layer(num_q_heads: int, num_kv_heads: int, head_dim: int,
                block_len, rank_k, rank_v=None, *, batch: int = 1,
                tail_lengths=None, seed: int = 0, layer: int = 0,
                device="cpu", q_scale: float = 1.0, basis: str = "random",
                poison_gaps: bool = False, tail_present: bool = True) -> LayerInputs:
    """Draw one layer's inputs for an explicit table.

    ``rank_k`` / ``rank_v`` are [num_blocks, num_kv_heads] (or flat).  ``basis``
    is "random" (orthonormal rows from QR) or "identity" (P = first r rows of
    the identity, exact in bf16)."""
    block_len = np.asarray(block_len, dtype=np.int32).reshape(-1)
    nb, hk, d = int(block_len.shape[0]), int(num_kv_heads), int(head_dim)
    rk = np.asarray(rank_k, dtype=np.int32).reshape(nb * hk)
    rv = rk.copy() if rank_v is None else np.asarray(rank_v, dtype=np.int32).reshape(nb * hk)
    gen = _torch_gen(device, seed, layer)
    gen_cpu = _torch_gen("cpu", seed + 104_729, layer)

    # element offsets, every factor 8-aligned, entries in (b, g) order
    offs = np.zeros((4, nb * hk), dtype=np.int64)
    cur = 0
    sizes = []
    for b in range(nb):
        for g in range(hk):
            e = b * hk + g
            for k, (rows, cols) in enumerate(((block_len[b], rk[e]), (rk[e], d),
                                              (block_len[b], rv[e]), (rv[e], d))):
                offs[k, e] = cur
                sz = int(rows) * int(cols)
                sizes.append((e, k, sz))
                cur += sz + ((-sz) % ALIGN)
    total = cur

    # draw factors grouped by (shape) so each group is one batched draw
    pieces = {}
    def group_draw(kind: str, ranks: np.ndarray):
        keys = {}
        for b in range(nb):
            for g in range(hk):
                e = b * hk + g
                shape = (int(block_len[b]), int(ranks[e])) if kind == "C" else (int(ranks[e]), d)
                keys.setdefault(shape, []).append(e)
        out = {}
        for shape in sorted(keys):
            es = keys[shape]
            m = len(es)
            if kind == "C":
                n, r = shape
                x = torch.randn((m, n, r), generator=gen, device=device, dtype=torch.float32)
                if r:
                    std = torch.rsqrt(torch.arange(1, r + 1, device=device, dtype=torch.float32))
                    x = x * std
            else:
                r, _ = shape
                if basis == "identity":
                    x = torch.eye(d, device=device, dtype=torch.float32)[:r].expand(m, r, d)
                elif r:
                    x = _orthonormal_rows(m, r, d, gen_cpu, device)
                else:
                    x = torch.zeros((m, 0, d), device=device)
            x = x.to(torch.bfloat16)
            for i, e in enumerate(es):
                out[e] = x[i].reshape(-1)
        return out

    ck, pk = group_draw("C", rk), group_draw("P", rk)
    cv, pv = group_draw("C", rv), group_draw("P", rv)
    fill = float("nan") if poison_gaps else 0.0
    parts = []
    for b in range(nb):
        for g in range(hk):
            e = b * hk + g
            for src in (ck, pk, cv, pv):
                t = src[e]
                parts.append(t)
                pad = (-int(t.numel())) % ALIGN
                if pad:
                    parts.append(torch.full((pad,), fill, device=device, dtype=torch.bfloat16))
    arena = torch.cat(parts) if parts else torch.zeros(0, device=device, dtype=torch.bfloat16)
    assert int(arena.numel()) == total

    q = torch.randn((batch, num_q_heads, d), generator=gen, device=device, dtype=torch.float32)
    q = (q * q_scale).to(torch.bfloat16)
    tl = np.zeros(batch, dtype=np.int64) if tail_lengths is None else np.asarray(tail_lengths, dtype=np.int64).reshape(batch)
    toff = np.zeros(batch + 1, dtype=np.int64)
    toff[1:] = np.cumsum(tl)
    ttot = int(toff[-1])
    if tail_present:
        tk = torch.randn((ttot, hk, d), generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
        tv = torch.randn((ttot, hk, d), generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
    else:
        tk = tv = None
    return LayerInputs(num_q_heads, hk, d, block_len, rk, rv, offs[0], offs[1],
                       offs[2], offs[3], arena, q, tk, tv, toff,
                       meta=dict(seed=seed, layer=layer, q_scale=q_scale,
                                 basis=basis, poison_gaps=poison_gaps))


def make_config_layer(cfg: Config, layer: int, device="cpu", q_scale: float = 1.0,
                      poison_gaps: bool = False) -> LayerInputs:
    """Inputs of layer ``layer`` of a named workload."""
    ranks = draw_ranks(cfg, layer)
    tl = draw_tail_lengths(cfg, layer)
    return build_layer(cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                       np.full(cfg.num_blocks, cfg.block_len), ranks,
                       batch=cfg.batch, tail_lengths=tl, seed=cfg.seed,
                       layer=layer, device=device, q_scale=q_scale,
                       poison_gaps=poison_gaps)


def make_random_case(*, num_q_heads, num_kv_heads, head_dim, block_lens,
                     rank_choices, batch=1, tail_lengths=None, seed=0,
                     device="cpu", separate_kv_ranks=True, q_scale=1.0,
                     basis="random", poison_gaps=False) -> LayerInputs:
    """A small case with ranks drawn from ``rank_choices`` (clipped to
    min(n_b, d)), optionally different for K and V."""
    rng = _np_rng(seed, 99)
    bl = np.asarray(block_lens, dtype=np.int32)
    nb = bl.shape[0]
    caps = np.minimum(bl[:, None], head_dim)
    rk = np.minimum(rng.choice(np.asarray(rank_choices), size=(nb, num_kv_heads)), caps)
    rv = np.minimum(rng.choice(np.asarray(rank_choices), size=(nb, num_kv_heads)), caps) if separate_kv_ranks else rk
    return build_layer(num_q_heads, num_kv_heads, head_dim, bl, rk, rv,
                       batch=batch, tail_lengths=tail_lengths, seed=seed,
                       device=device, q_scale=q_scale, basis=basis,
                       poison_gaps=poison_gaps)


def make_dense_kv(block_lens, num_kv_heads: int, head_dim: int, *, seed: int = 0,
                  device="cpu", noise: float = 0.0, zero_blocks=()):
    """Dense keys and values of a prefix, the input of the compression stage:
    bf16 [sum(block_lens), num_kv_heads, head_dim] each (token-major, as a KV
    cache holds them).

    Recipe: for every block b and KV head g, independently for K and V,
    X = Z diag(s) Q + noise W with Z, W standard Gaussian [n_b, d], s_j =
    j^(-1/2) (variance 1/j, the decay law of the factor workloads) and Q an
    orthonormal d x d matrix (drawn and factorised on the host), so that X's
    singular values decay like sqrt(n_b / j).  Blocks listed in
    ``zero_blocks`` are all zeros (every singular value 0)."""
    bl = np.asarray(block_lens, dtype=np.int64).reshape(-1)
    nb, hk, d = int(bl.shape[0]), int(num_kv_heads), int(head_dim)
    gen = _torch_gen(device, seed, 7777)
    gen_cpu = _torch_gen("cpu", seed + 104_729, 7777)
    N = int(bl.sum())
    out = []
    s = torch.arange(1, d + 1, dtype=torch.float32, device=device).rsqrt()
    for _side in range(2):
        X = torch.empty((N, hk, d), dtype=torch.float32, device=device)
        Q = _orthonormal_rows(nb * hk, d, d, gen_cpu, device)  # [nb * hk, d, d]
        t0 = 0
        for b in range(nb):
            n = int(bl[b])
            for g in range(hk):
                if b in zero_blocks:
                    X[t0:t0 + n, g] = 0.0
                    continue
                Z = torch.randn((n, d), generator=gen, device=device)
                x = (Z * s) @ Q[b * hk + g]
                if noise:
                    x = x + noise * torch.randn((n, d), generator=gen, device=device)
                X[t0:t0 + n, g] = x
            t0 += n
        out.append(X.to(torch.bfloat16))
    return out[0], out[1]
