"""Python binding of libmilo (include/milo.h): argument marshalling only.

Every computation runs inside libmilo's CUDA kernels; this module converts
numpy arrays and torch tensors into the pointers and sizes the C ABI takes.
Importing it does not build anything: call ``paper_2609_29913_gb300.build``
(or ``__graft_entry__.build()``) first.  A missing library raises
:class:`MiloError` -- there is no fallback.

Functions carry the C names.  :class:`Prefix` is the convenience wrapper a
user calls: create once per layer from a block table, then ``decode`` per
step (torch tensors in, fp32 attention output out).
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libmilo.so")

MILO_OK = 0
STATUS_NAMES = {0: "MILO_OK", 1: "MILO_ERR_INVALID_ARG", 2: "MILO_ERR_BAD_TABLE",
                3: "MILO_ERR_ALIGNMENT", 4: "MILO_ERR_UNSUPPORTED", 5: "MILO_ERR_CUDA",
                6: "MILO_ERR_TIMEOUT", 7: "MILO_ERR_DEVICE_BOUNDS", 8: "MILO_ERR_WORKSPACE"}

# every symbol include/milo.h declares
EXPORTS = ["milo_status_string", "milo_version", "milo_last_error_message",
           "milo_validate_table", "milo_packed_layout", "milo_partition_prefix",
           "milo_chunk_prefix", "milo_prefix_create", "milo_prefix_destroy", "milo_prefix_get_info",
           "milo_workspace_size", "milo_attn_decode", "milo_attn_decode_static",
           "milo_get_device_status", "milo_call_info", "milo_tensor_min_rows",
           "milo_prefix_set_tensor_min_rows",
           "milo_attn_decode_reconstruct", "milo_prefix_set_rope", "milo_check_bounded_wait",
           "milo_encode_layout", "milo_encode_workspace_size", "milo_encode",
           "milo_prefix_offload", "milo_prefix_stage", "milo_quantize_int8", "milo_dequantize_int8",
           "milo_prefix_quantize_int8", "milo_prefix_storage_bytes"]

PATH_NAMES = {0: "chunks", 1: "tensor"}


class MiloError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str = ""):
        self.status = int(status)
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}" + (f" ({detail})" if detail else ""))


class BlockTableC(ctypes.Structure):
    _fields_ = [("num_blocks", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32),
                ("block_len", ctypes.c_void_p), ("rank_k", ctypes.c_void_p),
                ("rank_v", ctypes.c_void_p), ("off_ck", ctypes.c_void_p),
                ("off_pk", ctypes.c_void_p), ("off_cv", ctypes.c_void_p),
                ("off_pv", ctypes.c_void_p), ("arena", ctypes.c_void_p),
                ("arena_elems", ctypes.c_int64)]


class CallInfoC(ctypes.Structure):
    _fields_ = [("path", ctypes.c_int32), ("kernels", ctypes.c_int32),
                ("row_tiles", ctypes.c_int32), ("blocks", ctypes.c_int32)]


class EncodeParamsC(ctypes.Structure):
    _fields_ = [("num_blocks", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("block_len", ctypes.c_void_p),
                ("r_min", ctypes.c_int32), ("r_max", ctypes.c_int32),
                ("budget_k", ctypes.c_int64), ("budget_v", ctypes.c_int64)]


class PrefixInfoC(ctypes.Structure):
    _fields_ = [("num_blocks", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("num_q_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("max_batch", ctypes.c_int32),
                ("prefix_tokens", ctypes.c_int64), ("logical_factor_bytes", ctypes.c_int64),
                ("packed_bytes", ctypes.c_int64), ("packed_arena", ctypes.c_void_p)]


_lib = None


def lib():
    """The loaded libmilo (raises MiloError if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise MiloError(5, "load libmilo", f"{LIB_PATH} missing; build it first")
        L = ctypes.CDLL(LIB_PATH)
        P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        L.milo_status_string.argtypes = [i32]
        L.milo_status_string.restype = ctypes.c_char_p
        L.milo_version.restype = i32
        L.milo_last_error_message.restype = ctypes.c_char_p
        L.milo_validate_table.argtypes = [P]
        L.milo_packed_layout.argtypes = [P, P, P]
        L.milo_partition_prefix.argtypes = [P, i32, i32, P, P, P, P, P, P, P]
        L.milo_chunk_prefix.argtypes = [P, i32, P, P, P, P]
        L.milo_prefix_create.argtypes = [P, i32, i32, P, P]
        L.milo_prefix_destroy.argtypes = [P]
        L.milo_prefix_get_info.argtypes = [P, P]
        L.milo_workspace_size.argtypes = [P, i32, i64, P]
        L.milo_attn_decode.argtypes = [P, P, i32, P, P, P, i64, i64, ctypes.c_float, P, P,
                                       ctypes.c_size_t, P]
        L.milo_attn_decode_static.argtypes = [P, P, i32, P, P, P, i64, i64, ctypes.c_float, P, P]
        L.milo_attn_decode_reconstruct.argtypes = [P, P, i32, P, P, P, i64, i64, ctypes.c_float, P, P,
                                                   ctypes.c_size_t, P]
        L.milo_prefix_set_rope.argtypes = [P, ctypes.c_double, P]
        L.milo_check_bounded_wait.argtypes = [P, i64, i32, P]
        L.milo_encode_layout.argtypes = [P, P, P]
        L.milo_encode_workspace_size.argtypes = [P, P]
        L.milo_encode.argtypes = [P, P, P, P, i64, P, P, P, P, ctypes.c_size_t, P]
        L.milo_prefix_offload.argtypes = [P]
        L.milo_prefix_stage.argtypes = [P, P, ctypes.c_size_t, P]
        L.milo_quantize_int8.argtypes = [P, i64, P, P, P]
        L.milo_dequantize_int8.argtypes = [P, P, i64, P, P]
        L.milo_prefix_quantize_int8.argtypes = [P, i32]
        L.milo_prefix_storage_bytes.argtypes = [P, P, P, P]
        L.milo_get_device_status.argtypes = [P, P, i32, P]
        L.milo_call_info.argtypes = [P, i32, i64, P]
        L.milo_tensor_min_rows.restype = i32
        L.milo_prefix_set_tensor_min_rows.argtypes = [P, i32]
        for name in ("milo_validate_table", "milo_packed_layout", "milo_partition_prefix",
                     "milo_chunk_prefix", "milo_prefix_create", "milo_prefix_destroy", "milo_prefix_get_info",
                     "milo_workspace_size", "milo_attn_decode", "milo_attn_decode_static",
                     "milo_get_device_status", "milo_call_info", "milo_attn_decode_reconstruct",
                     "milo_prefix_set_tensor_min_rows",
                     "milo_prefix_set_rope", "milo_check_bounded_wait", "milo_encode_layout",
                     "milo_encode_workspace_size", "milo_encode", "milo_prefix_offload", "milo_prefix_stage",
                     "milo_quantize_int8", "milo_dequantize_int8", "milo_prefix_quantize_int8",
                     "milo_prefix_storage_bytes"):
            getattr(L, name).restype = i32
        _lib = L
    return _lib


def _check(status: int, where: str):
    if status != MILO_OK:
        detail = lib().milo_last_error_message().decode(errors="replace")
        raise MiloError(status, where, detail)


def _arr(a, dtype):
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


class HostTable:
    """Host-side arrays of a block table plus the device arena pointer, kept
    alive for as long as the ctypes struct built from them is used."""

    def __init__(self, *, num_kv_heads, head_dim, block_len, rank_k, rank_v, off_ck,
                 off_pk, off_cv, off_pv, arena_ptr=0, arena_elems=0):
        self.block_len = _arr(block_len, np.int32)
        self.rank_k = _arr(rank_k, np.int32)
        self.rank_v = _arr(rank_v, np.int32)
        self.off_ck = _arr(off_ck, np.int64)
        self.off_pk = _arr(off_pk, np.int64)
        self.off_cv = _arr(off_cv, np.int64)
        self.off_pv = _arr(off_pv, np.int64)
        nb = int(self.block_len.shape[0])
        ptr = lambda a: a.ctypes.data if a.size else None
        self.c = BlockTableC(nb, int(num_kv_heads), int(head_dim), ptr(self.block_len),
                             ptr(self.rank_k), ptr(self.rank_v), ptr(self.off_ck),
                             ptr(self.off_pk), ptr(self.off_cv), ptr(self.off_pv),
                             int(arena_ptr) or None, int(arena_elems))

    @property
    def num_entries(self) -> int:
        return int(self.c.num_blocks) * int(self.c.num_kv_heads)

    @classmethod
    def from_layer(cls, layer):
        """From a ``workloads.LayerInputs`` (arena on the GPU)."""
        return cls(**layer.table_arrays(), arena_ptr=layer.arena.data_ptr(),
                   arena_elems=int(layer.arena.numel()))


def milo_validate_table(table: HostTable) -> int:
    return int(lib().milo_validate_table(ctypes.byref(table.c)))


def milo_packed_layout(table: HostTable):
    offs = np.zeros(max(table.num_entries * 4, 1), dtype=np.int64)
    total = ctypes.c_int64(0)
    _check(lib().milo_packed_layout(ctypes.byref(table.c), offs.ctypes.data, ctypes.byref(total)),
           "milo_packed_layout")
    return offs[:table.num_entries * 4].reshape(-1, 4), int(total.value)


def milo_partition_prefix(table: HostTable, num_shares: int) -> dict:
    """The tensor-core grid's partition over num_shares shares: entry, t0, t1,
    slot per segment, share_begin, num_slots."""
    nseg, nslot = ctypes.c_int32(0), ctypes.c_int32(0)
    L = lib()
    _check(L.milo_partition_prefix(ctypes.byref(table.c), int(num_shares), 0, None, None, None,
                                   None, None, ctypes.byref(nseg), ctypes.byref(nslot)),
           "milo_partition_prefix")
    n = int(nseg.value)
    out = {k: np.zeros(max(n, 1), dtype=np.int32) for k in ("entry", "t0", "t1", "slot")}
    sb = np.zeros(int(num_shares) + 1, dtype=np.int32)
    _check(L.milo_partition_prefix(ctypes.byref(table.c), int(num_shares), n,
                                   out["entry"].ctypes.data, out["t0"].ctypes.data,
                                   out["t1"].ctypes.data, out["slot"].ctypes.data,
                                   sb.ctypes.data, None, None), "milo_partition_prefix")
    res = {k: v[:n] for k, v in out.items()}
    res["share_begin"] = sb
    res["num_slots"] = int(nslot.value)
    return res


def milo_chunk_prefix(table: HostTable) -> dict:
    """The chunk grid's work list: entry, t0, t1 per chunk."""
    n = ctypes.c_int32(0)
    L = lib()
    _check(L.milo_chunk_prefix(ctypes.byref(table.c), 0, None, None, None, ctypes.byref(n)),
           "milo_chunk_prefix")
    k = int(n.value)
    out = {key: np.zeros(max(k, 1), dtype=np.int32) for key in ("entry", "t0", "t1")}
    _check(L.milo_chunk_prefix(ctypes.byref(table.c), k, out["entry"].ctypes.data, out["t0"].ctypes.data,
                               out["t1"].ctypes.data, None), "milo_chunk_prefix")
    return {key: v[:k] for key, v in out.items()}


def _stream_ptr(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


def milo_prefix_create(table: HostTable, num_q_heads: int, max_batch: int, stream=None) -> int:
    plan = ctypes.c_void_p(0)
    _check(lib().milo_prefix_create(ctypes.byref(table.c), int(num_q_heads), int(max_batch),
                                    _stream_ptr(stream), ctypes.byref(plan)), "milo_prefix_create")
    return int(plan.value)


def milo_prefix_destroy(plan: int) -> None:
    _check(lib().milo_prefix_destroy(plan), "milo_prefix_destroy")


def milo_prefix_get_info(plan: int) -> dict:
    info = PrefixInfoC()
    _check(lib().milo_prefix_get_info(plan, ctypes.byref(info)), "milo_prefix_get_info")
    return {name: getattr(info, name) for name, _ in PrefixInfoC._fields_}


def milo_workspace_size(plan: int, batch: int, max_tail_tokens: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().milo_workspace_size(plan, int(batch), int(max_tail_tokens), ctypes.byref(n)),
           "milo_workspace_size")
    return int(n.value)


def milo_call_info(plan: int, batch: int, max_tail_tokens: int) -> dict:
    """How a call of this shape runs: path (0 chunks, 1 tensor),
    kernels per call, row tiles and main-grid blocks (host only)."""
    info = CallInfoC()
    _check(lib().milo_call_info(plan, int(batch), int(max_tail_tokens), ctypes.byref(info)),
           "milo_call_info")
    return {name: getattr(info, name) for name, _ in CallInfoC._fields_}


def milo_tensor_min_rows() -> int:
    return int(lib().milo_tensor_min_rows())


def milo_attn_decode(plan: int, q_ptr: int, batch: int, tail_k_ptr: int, tail_v_ptr: int,
                     tail_offsets_ptr: int, tail_rows: int, max_tail_tokens: int,
                     softmax_scale: float, out_ptr: int, workspace_ptr: int,
                     workspace_bytes: int, stream=None) -> None:
    _check(lib().milo_attn_decode(plan, q_ptr, int(batch), tail_k_ptr or None, tail_v_ptr or None,
                                  tail_offsets_ptr or None, int(tail_rows), int(max_tail_tokens),
                                  float(softmax_scale), out_ptr, workspace_ptr,
                                  int(workspace_bytes), _stream_ptr(stream)), "milo_attn_decode")


def milo_attn_decode_static(plan: int, q_ptr: int, batch: int, tail_k_ptr: int, tail_v_ptr: int,
                            tail_offsets_ptr: int, tail_rows: int, max_tail_tokens: int,
                            softmax_scale: float, out_ptr: int, stream=None) -> None:
    """milo_attn_decode with the library's built-in scratch (no workspace)."""
    _check(lib().milo_attn_decode_static(plan, q_ptr, int(batch), tail_k_ptr or None,
                                         tail_v_ptr or None, tail_offsets_ptr or None,
                                         int(tail_rows), int(max_tail_tokens), float(softmax_scale),
                                         out_ptr, _stream_ptr(stream)), "milo_attn_decode_static")


def milo_attn_decode_reconstruct(plan: int, q_ptr: int, batch: int, tail_k_ptr: int, tail_v_ptr: int,
                                 tail_offsets_ptr: int, tail_rows: int, max_tail_tokens: int,
                                 softmax_scale: float, out_ptr: int, workspace_ptr: int,
                                 workspace_bytes: int, stream=None) -> None:
    """The same call by reconstruct-then-attend (the paper's own path)."""
    _check(lib().milo_attn_decode_reconstruct(plan, q_ptr, int(batch), tail_k_ptr or None, tail_v_ptr or None,
                                              tail_offsets_ptr or None, int(tail_rows), int(max_tail_tokens),
                                              float(softmax_scale), out_ptr, workspace_ptr,
                                              int(workspace_bytes), _stream_ptr(stream)),
           "milo_attn_decode_reconstruct")


def milo_prefix_set_rope(plan: int, rope_theta: float, block_pos=None) -> None:
    """Declare the plan's factors pre-RoPE (rope_theta > 0) or not (0);
    block_pos: one int64 position per block, or None for the concatenated
    prefix."""
    pos = None if block_pos is None else _arr(block_pos, np.int64)
    _check(lib().milo_prefix_set_rope(plan, float(rope_theta), None if pos is None else pos.ctypes.data),
           "milo_prefix_set_rope")


def milo_check_bounded_wait(plan: int, limit_ns: int, arrive: bool, stream=None) -> None:
    """One warp's bounded wait on an mbarrier nothing completes (arrive=False)
    or that it completes itself; a wait that runs out sets MILO_ERR_TIMEOUT in
    the plan's status word."""
    _check(lib().milo_check_bounded_wait(plan, int(limit_ns), int(bool(arrive)), _stream_ptr(stream)),
           "milo_check_bounded_wait")


def _encode_params(block_len, num_kv_heads, head_dim, r_min, r_max, budget_k, budget_v):
    bl = _arr(block_len, np.int32)
    c = EncodeParamsC(int(bl.shape[0]), int(num_kv_heads), int(head_dim), bl.ctypes.data if bl.size else None,
                      int(r_min), int(r_max), int(budget_k), int(budget_v))
    return c, bl


def milo_encode_layout(block_len, num_kv_heads, head_dim, r_max, r_min=0, budget_k=None, budget_v=None):
    """Element offsets [E][4] of C^K, P^K, C^V, P^V and the element count of
    the arena milo_encode fills."""
    big = 1 << 62
    c, bl = _encode_params(block_len, num_kv_heads, head_dim, r_min, r_max,
                           big if budget_k is None else budget_k, big if budget_v is None else budget_v)
    E = int(bl.shape[0]) * int(num_kv_heads)
    offs = np.zeros((max(E, 1), 4), dtype=np.int64)
    n = ctypes.c_int64(0)
    _check(lib().milo_encode_layout(ctypes.byref(c), offs.ctypes.data, ctypes.byref(n)), "milo_encode_layout")
    return offs[:E], int(n.value)


def encode(k, v, block_len, *, r_min, r_max, budget_k, budget_v, stream=None):
    """Compress a prefix on the GPU (milo_encode).  k, v: bf16 cuda tensors
    [sum(block_len), Hkv, d].  Returns a dict: ``arena`` (bf16 cuda tensor),
    ``rank_k``, ``rank_v`` (numpy int32 [E]), the four offset arrays,
    ``sigma`` (fp32 cuda tensor [2E, d]) and the table arguments, ready for
    :class:`HostTable` (``HostTable(**table_args(result))``)."""
    import torch
    N, hkv, d = (int(x) for x in k.shape)
    bl = _arr(block_len, np.int32)
    if int(bl.sum()) != N or tuple(v.shape) != tuple(k.shape):
        raise ValueError("k, v must be [sum(block_len), Hkv, d]")
    c, bl = _encode_params(bl, hkv, d, r_min, r_max, budget_k, budget_v)
    E = int(bl.shape[0]) * hkv
    offs, n = milo_encode_layout(bl, hkv, d, r_max, r_min, budget_k, budget_v)
    wsb = ctypes.c_size_t(0)
    L = lib()
    _check(L.milo_encode_workspace_size(ctypes.byref(c), ctypes.byref(wsb)), "milo_encode_workspace_size")
    dev = k.device
    arena = torch.zeros(max(n, 8), dtype=torch.bfloat16, device=dev)
    ranks = torch.zeros((2, max(E, 1)), dtype=torch.int32, device=dev)
    sigma = torch.zeros((2 * E, d), dtype=torch.float32, device=dev)
    ws = torch.empty(int(wsb.value) + 256, dtype=torch.uint8, device=dev)
    wp = (ws.data_ptr() + 255) // 256 * 256
    _check(L.milo_encode(ctypes.byref(c), k.data_ptr(), v.data_ptr(), arena.data_ptr(), int(arena.numel()),
                         ranks[0].data_ptr(), ranks[1].data_ptr(), sigma.data_ptr(), wp, int(wsb.value),
                         _stream_ptr(stream)), "milo_encode")
    rk = ranks.cpu().numpy()
    return dict(arena=arena, rank_k=rk[0, :E].copy(), rank_v=rk[1, :E].copy(), off_ck=offs[:, 0].copy(),
                off_pk=offs[:, 1].copy(), off_cv=offs[:, 2].copy(), off_pv=offs[:, 3].copy(), sigma=sigma,
                block_len=bl.copy(), num_kv_heads=hkv, head_dim=d)


def table_args(enc: dict) -> dict:
    """HostTable arguments of an :func:`encode` result."""
    return dict(num_kv_heads=enc["num_kv_heads"], head_dim=enc["head_dim"], block_len=enc["block_len"],
                rank_k=enc["rank_k"], rank_v=enc["rank_v"], off_ck=enc["off_ck"], off_pk=enc["off_pk"],
                off_cv=enc["off_cv"], off_pv=enc["off_pv"], arena_ptr=enc["arena"].data_ptr(),
                arena_elems=int(enc["arena"].numel()))


def milo_quantize_int8(packed, codes, params, stream=None) -> None:
    """INT8 codes and group parameters of a packed arena (cuda uint8 tensors:
    ``packed`` of B bytes, ``codes`` of B/2, ``params`` of B/32)."""
    nbytes = packed.numel() * packed.element_size()
    if codes.numel() * codes.element_size() < nbytes // 2 or params.numel() * params.element_size() < nbytes // 32:
        raise ValueError("codes or params too small")
    _check(lib().milo_quantize_int8(packed.data_ptr(), nbytes, codes.data_ptr(), params.data_ptr(),
                                    _stream_ptr(stream)), "milo_quantize_int8")


def milo_dequantize_int8(codes, params, packed, stream=None) -> None:
    """The bf16 values read back from INT8 codes into ``packed`` (B bytes)."""
    nbytes = packed.numel() * packed.element_size()
    if codes.numel() * codes.element_size() < nbytes // 2 or params.numel() * params.element_size() < nbytes // 32:
        raise ValueError("codes or params too small")
    _check(lib().milo_dequantize_int8(codes.data_ptr(), params.data_ptr(), nbytes, packed.data_ptr(),
                                      _stream_ptr(stream)), "milo_dequantize_int8")


def milo_prefix_storage_bytes(plan: int) -> dict:
    b, q, h = ctypes.c_int64(0), ctypes.c_int32(0), ctypes.c_int32(0)
    _check(lib().milo_prefix_storage_bytes(plan, ctypes.byref(b), ctypes.byref(q), ctypes.byref(h)),
           "milo_prefix_storage_bytes")
    return {"bytes": b.value, "int8": bool(q.value), "on_host": bool(h.value)}


def milo_get_device_status(plan: int, stream=None, clear: bool = False) -> int:
    code = ctypes.c_int32(0)
    _check(lib().milo_get_device_status(plan, _stream_ptr(stream), int(bool(clear)),
                                        ctypes.byref(code)), "milo_get_device_status")
    return int(code.value)


class Prefix:
    """One layer's compressed prefix on the GPU (a libmilo plan).

    ``Prefix(table, num_q_heads, max_batch)`` packs the factors; ``decode``
    runs one attention call into a preallocated fp32 output."""

    def __init__(self, table: HostTable, num_q_heads: int, max_batch: int, stream=None):
        self.table = table
        self.num_q_heads = int(num_q_heads)
        self.max_batch = int(max_batch)
        self.head_dim = int(table.c.head_dim)
        self.num_kv_heads = int(table.c.num_kv_heads)
        self.plan = milo_prefix_create(table, num_q_heads, max_batch, stream)
        self.info = milo_prefix_get_info(self.plan)

    @classmethod
    def from_layer(cls, layer, max_batch=None, stream=None):
        return cls(HostTable.from_layer(layer), layer.num_q_heads,
                   max_batch or layer.batch, stream)

    def workspace_size(self, batch: int, max_tail_tokens: int) -> int:
        return milo_workspace_size(self.plan, batch, max_tail_tokens)

    def set_rope(self, rope_theta: float, block_pos=None) -> None:
        """The factors are those of pre-RoPE keys (see milo_prefix_set_rope);
        decode_reconstruct then rotates the reconstructed keys."""
        milo_prefix_set_rope(self.plan, rope_theta, block_pos)

    def decode_reconstruct(self, q, tail_k=None, tail_v=None, tail_offsets=None, max_tail_tokens=0,
                           softmax_scale: float = 0.0, out=None, workspace=None, stream=None):
        """``decode`` by reconstruct-then-attend (milo_attn_decode_reconstruct)."""
        return self.decode(q, tail_k, tail_v, tail_offsets, max_tail_tokens, softmax_scale, out, workspace,
                           stream, _call=milo_attn_decode_reconstruct)

    def decode(self, q, tail_k=None, tail_v=None, tail_offsets=None, max_tail_tokens=0,
               softmax_scale: float = 0.0, out=None, workspace=None, stream=None, _call=None):
        """q: bf16 [batch, Hq, d] cuda tensor; tails bf16 [rows, Hkv, d];
        tail_offsets int64 cuda tensor [batch + 1].  Returns fp32 out."""
        import torch
        batch = int(q.shape[0])
        made = []  # buffers allocated here, on torch's current stream
        if out is None:
            out = torch.empty((batch, self.num_q_heads, self.head_dim), device=q.device,
                              dtype=torch.float32)
            made.append(out)
        need = self.workspace_size(batch, max_tail_tokens)
        if workspace is None:
            workspace = torch.empty(need, device=q.device, dtype=torch.uint8)
            made.append(workspace)
        tail_rows = int(tail_k.shape[0]) if (tail_k is not None and max_tail_tokens > 0) else 0
        (_call or milo_attn_decode)(self.plan, q.data_ptr(), batch,
                                    tail_k.data_ptr() if tail_rows else 0,
                                    tail_v.data_ptr() if tail_rows else 0,
                                    tail_offsets.data_ptr() if tail_rows else 0,
                                    tail_rows, max_tail_tokens if tail_rows else 0, softmax_scale,
                                    out.data_ptr(), workspace.data_ptr(),
                                    workspace.numel() * workspace.element_size(), stream)
        if isinstance(stream, torch.cuda.Stream):
            # the call runs on `stream`: keep the caching allocator from
            # handing these buffers out again before it has finished
            for t in made:
                t.record_stream(stream)
        return out

    def set_tensor_min_rows(self, rows: int) -> None:
        """Calls with at least ``rows`` query rows per KV head take the
        tensor-core path (milo_prefix_set_tensor_min_rows)."""
        _check(lib().milo_prefix_set_tensor_min_rows(self.plan, int(rows)), "milo_prefix_set_tensor_min_rows")

    def offload(self) -> None:
        """Move the packed arena to pinned host memory (milo_prefix_offload)."""
        _check(lib().milo_prefix_offload(self.plan), "milo_prefix_offload")
        self.info = milo_prefix_get_info(self.plan)

    def quantize_int8(self, to_host: bool = False) -> None:
        """Hold the arena as INT8 codes (milo_prefix_quantize_int8), in device
        memory or, with ``to_host``, in mapped pinned host memory."""
        _check(lib().milo_prefix_quantize_int8(self.plan, int(bool(to_host))), "milo_prefix_quantize_int8")
        self.info = milo_prefix_get_info(self.plan)

    def storage(self) -> dict:
        """Bytes of the arena at rest, whether INT8, whether on the host."""
        return milo_prefix_storage_bytes(self.plan)

    def stage(self, buffer, stream=None) -> None:
        """Enqueue the copy (an offloaded plan) or the dequantisation (an INT8
        plan) of the arena into ``buffer`` (a cuda uint8 tensor of at least
        info['packed_bytes'] bytes) on ``stream``; the following decode calls
        read it there.  ``buffer`` None: an INT8 plan in device memory goes
        back to reading its codes directly."""
        if buffer is None:
            _check(lib().milo_prefix_stage(self.plan, None, 0, _stream_ptr(stream)), "milo_prefix_stage")
            self.info = milo_prefix_get_info(self.plan)
            return
        _check(lib().milo_prefix_stage(self.plan, buffer.data_ptr(), buffer.numel() * buffer.element_size(),
                                       _stream_ptr(stream)), "milo_prefix_stage")

    def status(self, stream=None, clear=False) -> int:
        return milo_get_device_status(self.plan, stream, clear)

    def close(self):
        if getattr(self, "plan", None):
            milo_prefix_destroy(self.plan)
            self.plan = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
