"""A compressed prefix at rest: the block table and its bf16 arena, in one
.npz file.

The low-rank cache is produced once by the compression stage (Alg. 1,
Stage 1: per block and KV head the truncated factors C^K, P^K, C^V, P^V of
Eq. 3 at the ranks of Eq. 7) and read by every decode step after it
(Stage 2).  Saving it lets a prefix be encoded once and served later, the
pre-encoded store the paper's pipeline keeps.  Host side only: the arena is
kept as bf16 bit patterns (uint16); `prefix_from_file` copies it to the
device and builds a plan with milo_prefix_create, which validates the table
(lengths, ranks, offsets and overlaps) before anything is launched.
"""
from __future__ import annotations

import numpy as np

FORMAT = "milo-prefix/1"
_INT32 = ("block_len", "rank_k", "rank_v")
_INT64 = ("off_ck", "off_pk", "off_cv", "off_pv")


def _bits(arena) -> np.ndarray:
    """bf16 bit patterns of `arena` (a uint16 / int16 array, or a bf16 tensor)."""
    if hasattr(arena, "detach"):
        import torch
        t = arena.detach().cpu().contiguous()
        if t.dtype != torch.bfloat16:
            raise ValueError("the arena tensor must be bf16")
        return t.view(torch.int16).numpy().view(np.uint16).reshape(-1)
    a = np.asarray(arena)
    if a.dtype not in (np.uint16, np.int16):
        raise ValueError("the arena must hold bf16 bit patterns (uint16)")
    return np.ascontiguousarray(a.view(np.uint16).reshape(-1))


def save_prefix(path, *, num_kv_heads, head_dim, block_len, rank_k, rank_v, off_ck, off_pk, off_cv, off_pv,
                arena) -> None:
    """Write the table (the arguments of milo_block_table_t, offsets in
    elements) and the arena to `path` (.npz, no pickled objects)."""
    fields = {k: np.ascontiguousarray(np.asarray(v), dtype=np.int32)
              for k, v in zip(_INT32, (block_len, rank_k, rank_v))}
    fields.update({k: np.ascontiguousarray(np.asarray(v), dtype=np.int64)
                   for k, v in zip(_INT64, (off_ck, off_pk, off_cv, off_pv))})
    np.savez(path, format=np.array(FORMAT), num_kv_heads=np.int32(num_kv_heads), head_dim=np.int32(head_dim),
             arena=_bits(arena), **fields)


def load_prefix(path) -> dict:
    """Read a file written by save_prefix: a dict of the table's fields and
    `arena` (uint16 bf16 bit patterns).  Raises ValueError for another
    format, a missing field, a wrong type or inconsistent lengths."""
    with np.load(path, allow_pickle=False) as z:
        names = set(z.files)
        need = {"format", "num_kv_heads", "head_dim", "arena", *_INT32, *_INT64}
        if not need <= names:
            raise ValueError(f"not a saved prefix: missing {sorted(need - names)}")
        if str(z["format"]) != FORMAT:
            raise ValueError(f"unknown prefix format {str(z['format'])!r}")
        out = {"num_kv_heads": int(z["num_kv_heads"]), "head_dim": int(z["head_dim"])}
        for k in _INT32:
            if z[k].dtype != np.int32 or z[k].ndim != 1:
                raise ValueError(f"{k}: expected a 1-D int32 array")
            out[k] = z[k].copy()
        for k in _INT64:
            if z[k].dtype != np.int64 or z[k].ndim != 1:
                raise ValueError(f"{k}: expected a 1-D int64 array")
            out[k] = z[k].copy()
        if z["arena"].dtype != np.uint16 or z["arena"].ndim != 1:
            raise ValueError("arena: expected a 1-D uint16 array")
        out["arena"] = z["arena"].copy()
    entries = out["block_len"].shape[0] * out["num_kv_heads"]
    for k in _INT32[1:] + _INT64:
        if out[k].shape[0] != entries:
            raise ValueError(f"{k}: {out[k].shape[0]} values for {entries} entries")
    return out


def prefix_from_file(path, num_q_heads: int, max_batch: int, stream=None):
    """A plan (milo.Prefix) on the current CUDA device from a saved prefix.
    The device copy of the arena is released once the plan has packed it."""
    import torch

    from . import milo
    d = load_prefix(path)
    arena = torch.from_numpy(d.pop("arena").view(np.int16)).to("cuda").view(torch.bfloat16)
    table = milo.HostTable(**d, arena_ptr=arena.data_ptr(), arena_elems=int(arena.numel()))
    pre = milo.Prefix(table, num_q_heads, max_batch, stream)
    # the plan holds its packed copy; the table no longer points at the arena
    table.c.arena = None
    table.c.arena_elems = 0
    del arena
    return pre
