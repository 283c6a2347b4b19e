"""Thin ctypes binding of libbudgetdraft (include/budgetdraft.h).

Argument marshalling only: every computation runs in the library's CUDA kernels.  torch
tensors provide device memory and the current CUDA stream.  There is no fallback: if
the library is not built, or an argument is rejected, these functions raise.
"""

from __future__ import annotations

import ctypes
import os

import torch

from .build import LIB_PATH

BD_OK = 0
BD_ERR_CUDA = -5
BD_OP_SELECT, BD_OP_DRAFT, BD_OP_VERIFY = 1, 2, 3
BD_DRAFT_VIEW_READY = 1
BD_SELECT_WINDOW_READY = 1
BD_DTYPE_BF16, BD_DTYPE_F32 = 1, 2


class BdShape(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("h_q", ctypes.c_int32), ("h_kv", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("t_ctx", ctypes.c_int32), ("t_cap", ctypes.c_int32),
                ("seq_lens", ctypes.c_void_p)]

    def __repr__(self):
        return (f"BdShape(batch={self.batch}, h_q={self.h_q}, h_kv={self.h_kv}, head_dim={self.head_dim}, "
                f"t_ctx={self.t_ctx}, t_cap={self.t_cap})")


class BudgetDraftError(RuntimeError):
    def __init__(self, func, status):
        self.status = status
        super().__init__(f"{func} failed: {bd_strerror(status)} ({status})")


_lib = None
_P = ctypes.c_void_p
_SHAPE = ctypes.POINTER(BdShape)
_SIGNATURES = {
    "bd_workspace_size": (ctypes.c_size_t, [_SHAPE, ctypes.c_int, ctypes.c_int, ctypes.c_int]),
    "bd_select_budget": (ctypes.c_int, [_SHAPE, _P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int, ctypes.c_int, ctypes.c_uint, _P, _P, _P, ctypes.c_size_t,
                                        _P]),
    "bd_draft_attn": (ctypes.c_int, [_SHAPE, _P, _P, _P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_uint, _P,
                                     _P, _P, ctypes.c_size_t, _P]),
    "bd_draft_attn_static": (ctypes.c_int, [_SHAPE, _P, _P, _P, _P, _P, ctypes.c_int, ctypes.c_int, _P, _P,
                                            _P]),
    "bd_draft_static_status": (ctypes.c_int, [_P]),
    "bd_verify_attn": (ctypes.c_int, [_SHAPE, _P, ctypes.c_int, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "bd_combine": (ctypes.c_int, [_P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P, _P, _P]),
    "bd_argmax": (ctypes.c_int, [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P, _P]),
    "bd_accept": (ctypes.c_int, [ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P]),
    "bd_advance": (ctypes.c_int, [_SHAPE, ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, _P, _P, _P, ctypes.c_int, _P,
                                  _P]),
    "bd_write_block_rows": (ctypes.c_int, [_SHAPE, ctypes.c_int, _P, _P, _P, _P, _P]),
    "bd_check_wait_timeout": (ctypes.c_int, [_P, ctypes.c_size_t, ctypes.c_int, _P]),
    "bd_workspace_status": (ctypes.c_int, [_P, _P]),
    "bd_strerror": (ctypes.c_char_p, [ctypes.c_int]),
}


def library():
    """Load libbudgetdraft.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run paper_2606_00144_gb300.build.build() first")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def exported_symbols():
    return list(_SIGNATURES)


def bd_strerror(status: int) -> str:
    return library().bd_strerror(int(status)).decode()


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(name, status):
    if status != BD_OK:
        raise BudgetDraftError(name, status)


def make_shape(batch, h_q, h_kv, head_dim, t_ctx, t_cap, seq_lens=None) -> BdShape:
    """seq_lens: optional int32 device tensor [batch] of per-sequence context lengths (t_ctx
    is then the longest); the tensor must outlive every call made with this shape."""
    return BdShape(int(batch), int(h_q), int(h_kv), int(head_dim), int(t_ctx), int(t_cap), _ptr(seq_lens))


def shape_of(k_cache: torch.Tensor, h_q: int, t_ctx: int) -> BdShape:
    b, h_kv, t_cap, d = k_cache.shape
    return make_shape(b, h_q, h_kv, d, t_ctx, t_cap)


def bd_workspace_size(shape: BdShape, op: int, budget: int, n_q: int) -> int:
    return int(library().bd_workspace_size(ctypes.byref(shape), op, int(budget), int(n_q)))


class Workspace:
    """A zero-filled device buffer sized for a set of operations (see bd_workspace_size)."""

    def __init__(self, nbytes: int, device=None):
        self.nbytes = int(max(nbytes, 512))
        self.buf = torch.zeros(self.nbytes, dtype=torch.uint8, device=device or "cuda")

    @classmethod
    def for_step(cls, shape: BdShape, budget: int, window: int, gamma: int, device=None):
        sizes = [bd_workspace_size(shape, BD_OP_SELECT, budget, window),
                 bd_workspace_size(shape, BD_OP_DRAFT, budget, gamma),
                 bd_workspace_size(shape, BD_OP_VERIFY, budget, gamma + 1)]
        # an op this shape does not support reports size 0 here and its status when called
        if max(sizes) == 0:
            raise BudgetDraftError("bd_workspace_size", -1)
        return cls(max(sizes), device)

    @property
    def ptr(self):
        return self.buf.data_ptr()

    def status(self, stream=None) -> int:
        return int(library().bd_workspace_status(self.ptr, _stream(stream)))


def bd_select_budget(shape, k_cache, q_window, window_lse, window, budget, n_sink, n_recent, chunk,
                     idx_out, count_out, ws: Workspace, stream=None, flags=0):
    st = library().bd_select_budget(ctypes.byref(shape), _ptr(k_cache), _ptr(q_window), _ptr(window_lse),
                                    int(window), int(budget), int(n_sink), int(n_recent), int(chunk),
                                    int(flags), _ptr(idx_out), _ptr(count_out), ws.ptr, ws.nbytes,
                                    _stream(stream))
    _check("bd_select_budget", st)


def bd_draft_attn(shape, q, k_cache, v_cache, idx, count, budget, step_j, o_out, lse_out,
                  ws: Workspace, stream=None, flags=0):
    st = library().bd_draft_attn(ctypes.byref(shape), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(idx),
                                 _ptr(count), int(budget), int(step_j), int(flags), _ptr(o_out), _ptr(lse_out),
                                 ws.ptr, ws.nbytes, _stream(stream))
    _check("bd_draft_attn", st)


def bd_draft_attn_static(shape, q, k_cache, v_cache, idx, count, budget, step_j, o_out, lse_out, stream=None):
    """bd_draft_attn for callers that cannot allocate device memory: no workspace; the
    library's own 4 MiB device array holds the scratch, shared by every call (calls must
    not overlap on the GPU; the first call on a device must precede any stream capture)."""
    st = library().bd_draft_attn_static(ctypes.byref(shape), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(idx),
                                        _ptr(count), int(budget), int(step_j), _ptr(o_out), _ptr(lse_out),
                                        _stream(stream))
    _check("bd_draft_attn_static", st)


def bd_draft_static_status(stream=None) -> int:
    """Reads and clears the device-side error word of bd_draft_attn_static's array."""
    st = library().bd_draft_static_status(_stream(stream))
    if st == BD_ERR_CUDA:
        _check("bd_draft_static_status", st)
    return int(st)


def bd_verify_attn(shape, q, n_q, k_cache, v_cache, o_out, lse_out, ws: Workspace, stream=None):
    st = library().bd_verify_attn(ctypes.byref(shape), _ptr(q), int(n_q), _ptr(k_cache), _ptr(v_cache),
                                  _ptr(o_out), _ptr(lse_out), ws.ptr, ws.nbytes, _stream(stream))
    _check("bd_verify_attn", st)


def bd_combine(o_part, lse_part, n_split, rows, head_dim, o_out, lse_out, stream=None):
    st = library().bd_combine(_ptr(o_part), _ptr(lse_part), int(n_split), int(rows), int(head_dim),
                              _ptr(o_out), _ptr(lse_out), _stream(stream))
    _check("bd_combine", st)


def bd_argmax(logits, ids_out, stream=None):
    """ids_out[r] = arg max of logits[r] (bf16 or fp32 [rows, vocab], int32 [rows])."""
    if logits.dtype == torch.bfloat16:
        dtype = BD_DTYPE_BF16
    elif logits.dtype == torch.float32:
        dtype = BD_DTYPE_F32
    else:
        raise TypeError(f"bd_argmax: logits must be bf16 or fp32, got {logits.dtype}")
    if logits.dim() != 2 or not logits.is_contiguous():
        raise ValueError("bd_argmax: logits must be a contiguous [rows, vocab] tensor")
    rows, vocab = logits.shape
    st = library().bd_argmax(_ptr(logits), dtype, int(rows), int(vocab), _ptr(ids_out), _stream(stream))
    _check("bd_argmax", st)


def bd_accept(draft_tokens, verify_tokens, n_accept_out, emit_out, stream=None):
    """Accepted prefix length and emitted tokens: draft_tokens int32 [gamma, batch] (pass-major),
    verify_tokens int32 [batch, gamma + 1]."""
    batch, g1 = verify_tokens.shape
    st = library().bd_accept(int(batch), int(g1 - 1), _ptr(draft_tokens), _ptr(verify_tokens), _ptr(n_accept_out),
                             _ptr(emit_out), _stream(stream))
    _check("bd_accept", st)


def bd_advance(shape, window, n_q, n_accept, q_verify, verify_lse, q_window, window_lse, idx=None, count=None,
               advance_out=None, stream=None):
    """Slides the observation window (and appends to the sparse view) after acceptance."""
    cap = int(idx.shape[-1]) if idx is not None else 0
    st = library().bd_advance(ctypes.byref(shape), int(window), int(n_q), _ptr(n_accept), _ptr(q_verify),
                              _ptr(verify_lse), _ptr(q_window), _ptr(window_lse), _ptr(idx), _ptr(count), cap,
                              _ptr(advance_out), _stream(stream))
    _check("bd_advance", st)


def bd_write_block_rows(shape, n_rows, k_rows, v_rows, k_cache, v_cache, stream=None):
    """Writes rows t_ctx .. t_ctx + n_rows - 1 of the caches from dense [b, h_kv, n_rows, d]
    buffers (device or pinned host memory)."""
    st = library().bd_write_block_rows(ctypes.byref(shape), int(n_rows), _ptr(k_rows), _ptr(v_rows), _ptr(k_cache),
                                       _ptr(v_cache), _stream(stream))
    _check("bd_write_block_rows", st)


def bd_check_wait_timeout(ws: Workspace, limit_us: int, stream=None):
    """Runs the bounded-wait error path once (see the header); read the result with
    bd_workspace_status."""
    _check("bd_check_wait_timeout", library().bd_check_wait_timeout(ws.ptr, ws.nbytes, int(limit_us), _stream(stream)))


def bd_workspace_status(ws: Workspace, stream=None) -> int:
    return ws.status(stream)
