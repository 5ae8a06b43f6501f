"""Thin Python binding of the PSC C ABI (include/psc.h): argument marshalling only.

Every function here converts its arguments (torch tensors -> device pointers,
torch streams -> cudaStream_t) and calls the library function of the same
name; all work runs in the library's CUDA kernels.  There is no fallback: if
``libpsc_gb300.so`` is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpsc_gb300.so")

PSC_F32, PSC_BF16 = 0, 1
ROW_OK, ROW_DONE, ROW_REJECTED, ROW_OVERFLOW, ROW_LIMIT = 0, 1, 2, 3, 4
STATUS_NAMES = {0: "PSC_OK", 1: "PSC_ERR_ARG", 2: "PSC_ERR_GRAMMAR", 3: "PSC_ERR_CONFLICT",
                4: "PSC_ERR_LEXER_AMBIGUOUS", 5: "PSC_ERR_LIMIT", 6: "PSC_ERR_OOM", 7: "PSC_ERR_CUDA",
                8: "PSC_ERR_IO"}

EXPORTED = ["psc_compile", "psc_destroy", "psc_last_error", "psc_info", "psc_state_init", "psc_state_reset",
            "psc_state_destroy", "psc_advance", "psc_fill_mask", "psc_apply_mask", "psc_fill_apply",
            "psc_argmax_masked", "psc_states_download", "psc_host_classify", "psc_host_mask_row",
            "psc_host_advance", "psc_fill_apply_noalloc", "psc_fill_apply_argmax", "psc_save", "psc_load",
            "psc_decode_step", "psc_decode_step_mask", "psc_decode_step_advance", "psc_state_copy",
            "psc_host_classify_bottom_up", "psc_state_faults", "psc_check_wait"]
NOALLOC_MAX_ROWS = 16384


class PscError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {message}")
        self.code = code


class Options(ctypes.Structure):
    _fields_ = [("max_states", ctypes.c_int64), ("max_mask_bytes", ctypes.c_int64),
                ("threads", ctypes.c_int32), ("host_only", ctypes.c_int32),
                ("global_tables", ctypes.c_int32), ("max_bottom_up_bytes", ctypes.c_int64),
                ("max_dense_classifier_bytes", ctypes.c_int64)]


class InfoT(ctypes.Structure):
    _fields_ = [("V", ctypes.c_int32), ("W", ctypes.c_int32), ("n_lexer_states", ctypes.c_int32),
                ("n_parser_states", ctypes.c_int32), ("n_terminals", ctypes.c_int32),
                ("n_classifier_states", ctypes.c_int32), ("n_masks", ctypes.c_int32), ("eos_id", ctypes.c_int32),
                ("classifier_bytes", ctypes.c_int64), ("mask_bytes", ctypes.c_int64),
                ("states_built", ctypes.c_int64), ("compile_seconds", ctypes.c_double),
                ("advance_table_bytes", ctypes.c_int64), ("device_timeouts", ctypes.c_int64),
                ("bottom_up_states", ctypes.c_int64), ("bottom_up_bytes", ctypes.c_int64),
                ("classifier_sparse", ctypes.c_int64), ("advance_tables_packed", ctypes.c_int64)]


_lib = None


def load(path: str = LIB_PATH):
    """Load the library (raises if it is missing: there is no other backend)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2608_03065_gb300.build.build()")
    lib = ctypes.CDLL(path)
    vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    sig = {
        "psc_compile": (i32, [ctypes.c_char_p, sz, vp, vp, i32, i32, vp, vp]),
        "psc_destroy": (None, [vp]),
        "psc_last_error": (ctypes.c_char_p, []),
        "psc_info": (i32, [vp, vp]),
        "psc_state_init": (i32, [vp, i32, i32, vp, vp]),
        "psc_state_reset": (i32, [vp, vp, i32, vp]),
        "psc_state_destroy": (None, [vp]),
        "psc_advance": (i32, [vp, vp, vp, i32, vp, vp]),
        "psc_fill_mask": (i32, [vp, vp, i32, vp, vp]),
        "psc_apply_mask": (i32, [vp, i32, i64, vp, i32, i32, vp]),
        "psc_fill_apply": (i32, [vp, vp, i32, vp, i32, i64, i32, vp, vp]),
        "psc_argmax_masked": (i32, [vp, vp, i32, vp, i32, i64, i32, vp, vp]),
        "psc_states_download": (i32, [vp, vp, vp, vp, vp, vp]),
        "psc_host_classify": (i32, [vp, i32, vp, i32, i32]),
        "psc_host_classify_bottom_up": (i32, [vp, i32, vp, i32, i32]),
        "psc_host_mask_row": (i32, [vp, i32, vp]),
        "psc_host_advance": (i32, [vp, vp, vp, vp, i32, vp, i32]),
        "psc_fill_apply_noalloc": (i32, [vp, vp, vp, vp, vp, i32, i32, vp, i32, i64, i32, vp, vp]),
        "psc_fill_apply_argmax": (i32, [vp, vp, i32, vp, i32, i64, i32, vp, vp, vp]),
        "psc_save": (i32, [vp, ctypes.c_char_p]),
        "psc_decode_step": (i32, [vp, vp, i32, vp, i32, i64, i32, vp, vp, vp, vp]),
        "psc_decode_step_mask": (i32, [vp, vp, i32, vp, i32, i64, i32, vp, vp]),
        "psc_state_copy": (i32, [vp, vp, vp]),
        "psc_decode_step_advance": (i32, [vp, vp, i32, vp, vp, vp]),
        "psc_load": (i32, [ctypes.c_char_p, vp, vp]),
        "psc_state_faults": (i32, [vp, vp, i32, vp]),
        "psc_check_wait": (i32, [vp, i32, vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _check(code: int):
    if code != 0:
        raise PscError(code, (load().psc_last_error() or b"").decode(errors="replace"))


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


def _ptr(t, dtype=None, name="tensor", n=None):
    """Device address of a tensor argument; n = the elements the call reads or
    writes (a smaller or non-contiguous tensor is refused before any launch)."""
    if t is None:
        return None
    if n is not None and (t.numel() < n or not t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous tensor of at least {n} elements")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must have dtype {dtype}, got {t.dtype}")
    return t.data_ptr()


def _dtype_code(t):
    import torch
    if t.dtype == torch.bfloat16:
        return PSC_BF16
    if t.dtype == torch.float32:
        return PSC_F32
    raise ValueError(f"logits must be bf16 or f32, got {t.dtype}")


def _row_stride(t):
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("logits must be a 2-D tensor with unit column stride")
    return t.stride(0)


@dataclass
class Info:
    V: int
    W: int
    n_lexer_states: int
    n_parser_states: int
    n_terminals: int
    n_classifier_states: int
    n_masks: int
    eos_id: int
    classifier_bytes: int
    mask_bytes: int
    states_built: int
    compile_seconds: float
    advance_table_bytes: int
    device_timeouts: int
    bottom_up_states: int
    bottom_up_bytes: int
    classifier_sparse: int
    advance_tables_packed: int


class Handle:
    """A compiled grammar x vocabulary (owns the device tables)."""

    def __init__(self, ptr: int, V: int):
        self.ptr = ptr
        self.V = V
        self.W = (V + 31) // 32

    def __del__(self):
        if getattr(self, "ptr", None) and _lib is not None:
            _lib.psc_destroy(self.ptr)
            self.ptr = None

    def info(self) -> Info:
        out = InfoT()
        _check(load().psc_info(self.ptr, ctypes.byref(out)))
        return Info(*[getattr(out, f) for f, _ in InfoT._fields_])

    # --- host-side inspection of the compiled tables
    def host_classify(self, q: int, stack, status: int = ROW_OK) -> int:
        st = np.ascontiguousarray(np.asarray(stack, dtype=np.uint16))
        return load().psc_host_classify(self.ptr, q, st.ctypes.data if len(st) else None, len(st), status)

    def host_classify_bottom_up(self, q: int, stack, status: int = ROW_OK) -> int:
        """The same mask id through the bottom-up classifier (-2: not built, or
        the stack is not a path of the LR automaton)."""
        st = np.ascontiguousarray(np.asarray(stack, dtype=np.uint16))
        return load().psc_host_classify_bottom_up(self.ptr, q, st.ctypes.data if len(st) else None, len(st),
                                                  status)

    def host_mask_row(self, mask_id: int) -> np.ndarray:
        row = np.zeros(self.W, dtype=np.uint32)
        _check(load().psc_host_mask_row(self.ptr, mask_id, row.ctypes.data))
        return row

    def host_advance(self, cfg: dict, token: int, cap: int = 256) -> dict:
        """cfg = {"q", "stack" (list), "status"}; returns the next configuration."""
        stack = np.zeros(cap, dtype=np.uint16)
        stack[:len(cfg["stack"])] = cfg["stack"]
        q = ctypes.c_int32(cfg["q"])
        depth = ctypes.c_int32(len(cfg["stack"]))
        status = ctypes.c_int32(cfg["status"])
        _check(load().psc_host_advance(self.ptr, ctypes.byref(q), stack.ctypes.data, ctypes.byref(depth), cap,
                                       ctypes.byref(status), int(token)))
        return {"q": q.value, "stack": stack[:depth.value].tolist(), "status": status.value}

    def host_initial(self) -> dict:
        return {"q": 0, "stack": [0], "status": ROW_OK}


class States:
    """A batch of device-resident parser configurations (owns its device arrays)."""

    def __init__(self, ptr: int, handle: Handle, B: int, cap: int):
        self.ptr = ptr
        self.handle = handle
        self.B = B
        self.cap = cap

    def __del__(self):
        if getattr(self, "ptr", None) and _lib is not None:
            _lib.psc_state_destroy(self.ptr)
            self.ptr = None


# ------------------------------------------------------------------- the ABI
def _tables(global_tables: bool, packed_tables: bool) -> int:
    if global_tables and packed_tables:
        raise ValueError("global_tables and packed_tables exclude each other")
    return 1 if global_tables else 2 if packed_tables else 0


def psc_compile(grammar: str, vocab: list[bytes] | tuple, eos_id: int, host_only: bool = False,
                threads: int = 0, max_states: int = 0, max_mask_bytes: int = 0,
                global_tables: bool = False, bottom_up: bool = True, max_bottom_up_bytes: int = 0,
                max_dense_classifier_bytes: int = 0, packed_tables: bool = False) -> Handle:
    """vocab: list of token byte strings, or (blob uint8 array, offsets int64[V+1]).
    bottom_up=False builds no bottom-up classifier (every stack is walked from the top);
    max_dense_classifier_bytes < 0 holds the classifier in the sparse layout;
    global_tables=True has the advance read its parser tables from global memory,
    packed_tables=True stages them in the packed layout even when the dense one fits."""
    if isinstance(vocab, tuple):
        blob, offs = vocab
        blob = np.ascontiguousarray(blob, dtype=np.uint8)
        offs = np.ascontiguousarray(offs, dtype=np.int64)
    else:
        offs = np.zeros(len(vocab) + 1, dtype=np.int64)
        offs[1:] = np.cumsum([len(t) for t in vocab])
        blob = np.frombuffer(b"".join(vocab), dtype=np.uint8).copy()
    if blob.size == 0:
        blob = np.zeros(1, dtype=np.uint8)
    V = len(offs) - 1
    opts = Options(max_states, max_mask_bytes, threads, 1 if host_only else 0, _tables(global_tables, packed_tables),
                   max_bottom_up_bytes if bottom_up else -1, max_dense_classifier_bytes)
    g = grammar.encode("utf-8")
    out = ctypes.c_void_p()
    _check(load().psc_compile(g, len(g), blob.ctypes.data, offs.ctypes.data, V, eos_id, ctypes.byref(opts),
                              ctypes.byref(out)))
    return Handle(out.value, V)


def psc_save(h: Handle, path: str):
    _check(load().psc_save(h.ptr, os.fsencode(path)))


def psc_load(path: str, host_only: bool = False, global_tables: bool = False, bottom_up: bool = True,
             packed_tables: bool = False) -> Handle:
    opts = Options(0, 0, 0, 1 if host_only else 0, _tables(global_tables, packed_tables), 0 if bottom_up else -1, 0)
    out = ctypes.c_void_p()
    _check(load().psc_load(os.fsencode(path), ctypes.byref(opts), ctypes.byref(out)))
    h = Handle(out.value, 0)
    h.V = h.info().V
    h.W = (h.V + 31) // 32
    return h


def psc_state_init(h: Handle, B: int, cap: int = 256, stream=None) -> States:
    out = ctypes.c_void_p()
    _check(load().psc_state_init(h.ptr, B, cap, _stream(stream), ctypes.byref(out)))
    return States(out.value, h, B, cap)


def psc_state_reset(st: States, rows=None, stream=None):
    import torch
    n = st.B if rows is None else rows.numel()
    _check(load().psc_state_reset(st.ptr, _ptr(rows, torch.int32, "rows", n), n, _stream(stream)))


def psc_state_copy(dst: States, src: States, stream=None):
    """dst's rows := src's rows (same handle, B and cap), on the device."""
    _check(load().psc_state_copy(dst.ptr, src.ptr, _stream(stream)))


def psc_advance(h: Handle, st: States, tokens, row_status=None, stream=None):
    import torch
    _check(load().psc_advance(h.ptr, st.ptr, _ptr(tokens, torch.int32, "tokens", st.B), st.B,
                              _ptr(row_status, torch.int32, "row_status", st.B), _stream(stream)))


def psc_fill_mask(h: Handle, st: States, bitmask, stream=None):
    import torch
    if bitmask.shape != (st.B, h.W) or not bitmask.is_contiguous():
        raise ValueError(f"bitmask must be a contiguous [{st.B}, {h.W}] tensor")
    _check(load().psc_fill_mask(h.ptr, st.ptr, st.B, _ptr(bitmask, torch.int32, "bitmask"), _stream(stream)))


def psc_apply_mask(logits, bitmask, B: int, V: int, stream=None):
    import torch
    W = (V + 31) // 32
    if bitmask.shape[0] < B or bitmask.shape[1] != W or not bitmask.is_contiguous():
        raise ValueError(f"bitmask must be a contiguous [B, {W}] tensor")
    if logits.shape[0] < B or logits.shape[1] < V:
        raise ValueError("logits are smaller than [B, V]")
    _check(load().psc_apply_mask(_ptr(logits, None, "logits"), _dtype_code(logits), _row_stride(logits),
                                 _ptr(bitmask, torch.int32, "bitmask"), B, V, _stream(stream)))


def psc_fill_apply(h: Handle, st: States, logits, bitmask_out=None, V: int | None = None, stream=None):
    import torch
    V = h.V if V is None else V
    if logits.shape[0] != st.B or logits.shape[1] < V:
        raise ValueError("logits must be [B, >=V]")
    if bitmask_out is not None and (bitmask_out.shape != (st.B, h.W) or not bitmask_out.is_contiguous()):
        raise ValueError("bitmask_out must be a contiguous [B, W] tensor")
    _check(load().psc_fill_apply(h.ptr, st.ptr, st.B, _ptr(logits, None, "logits"), _dtype_code(logits),
                                 _row_stride(logits), V, _ptr(bitmask_out, torch.int32, "bitmask_out"),
                                 _stream(stream)))


def psc_argmax_masked(h: Handle, st: States, logits, tokens, stream=None):
    import torch
    if tokens.numel() != st.B:
        raise ValueError("tokens must hold B int32 values")
    _check(load().psc_argmax_masked(h.ptr, st.ptr, st.B, _ptr(logits, None, "logits"), _dtype_code(logits),
                                    _row_stride(logits), h.V, _ptr(tokens, torch.int32, "tokens", st.B),
                                    _stream(stream)))


def psc_fill_apply_argmax(h: Handle, st: States, logits, tokens, bitmask_out=None, stream=None):
    import torch
    if logits.shape[0] != st.B or logits.shape[1] < h.V:
        raise ValueError("logits must be [B, >=V]")
    if tokens.numel() != st.B:
        raise ValueError("tokens must hold B int32 values")
    if bitmask_out is not None and (bitmask_out.shape != (st.B, h.W) or not bitmask_out.is_contiguous()):
        raise ValueError("bitmask_out must be a contiguous [B, W] tensor")
    _check(load().psc_fill_apply_argmax(h.ptr, st.ptr, st.B, _ptr(logits, None, "logits"), _dtype_code(logits),
                                        _row_stride(logits), h.V, _ptr(bitmask_out, torch.int32, "bitmask_out"),
                                        _ptr(tokens, torch.int32, "tokens", st.B), _stream(stream)))


def psc_decode_step(h: Handle, st: States, logits, tokens, bitmask_out=None, row_status=None, stream=None):
    import torch
    if logits.shape[0] != st.B or logits.shape[1] < h.V:
        raise ValueError("logits must be [B, >=V]")
    if tokens.numel() != st.B:
        raise ValueError("tokens must hold B int32 values")
    if bitmask_out is not None and (bitmask_out.shape != (st.B, h.W) or not bitmask_out.is_contiguous()):
        raise ValueError("bitmask_out must be a contiguous [B, W] tensor")
    _check(load().psc_decode_step(h.ptr, st.ptr, st.B, _ptr(logits, None, "logits"), _dtype_code(logits),
                                  _row_stride(logits), h.V, _ptr(bitmask_out, torch.int32, "bitmask_out"),
                                  _ptr(tokens, torch.int32, "tokens", st.B),
                                  _ptr(row_status, torch.int32, "row_status", st.B), _stream(stream)))


def psc_decode_step_mask(h: Handle, st: States, logits, bitmask_out=None, stream=None):
    """First half of psc_decode_step: masking pass, greedy choices kept in the states."""
    import torch
    if logits.shape[0] != st.B or logits.shape[1] < h.V:
        raise ValueError("logits must be [B, >=V]")
    if bitmask_out is not None and (bitmask_out.shape != (st.B, h.W) or not bitmask_out.is_contiguous()):
        raise ValueError("bitmask_out must be a contiguous [B, W] tensor")
    _check(load().psc_decode_step_mask(h.ptr, st.ptr, st.B, _ptr(logits, None, "logits"), _dtype_code(logits),
                                       _row_stride(logits), h.V, _ptr(bitmask_out, torch.int32, "bitmask_out"),
                                       _stream(stream)))


def psc_decode_step_advance(h: Handle, st: States, tokens, row_status=None, stream=None):
    """Second half of psc_decode_step: tokens out, rows advanced and classified."""
    import torch
    if tokens.numel() != st.B:
        raise ValueError("tokens must hold B int32 values")
    _check(load().psc_decode_step_advance(h.ptr, st.ptr, st.B, _ptr(tokens, torch.int32, "tokens", st.B),
                                          _ptr(row_status, torch.int32, "row_status", st.B), _stream(stream)))


def psc_state_faults(st: States, reset: bool = False, stream=None) -> int:
    """Bounded in-kernel waits on these states that gave up (synchronises the stream)."""
    out = ctypes.c_int32(0)
    _check(load().psc_state_faults(st.ptr, ctypes.byref(out), 1 if reset else 0, _stream(stream)))
    return out.value


def psc_check_wait(st: States, limit: int = 4096, stream=None):
    """Self-test of fault reporting: a bounded wait that nothing completes gives up
    after `limit` polls and is counted on the states object."""
    _check(load().psc_check_wait(st.ptr, limit, _stream(stream)))


def psc_states_download(st: States, stream=None) -> dict:
    q = np.zeros(st.B, dtype=np.int32)
    depth = np.zeros(st.B, dtype=np.int32)
    stack = np.zeros((st.B, st.cap), dtype=np.uint16)
    status = np.zeros(st.B, dtype=np.int32)
    _check(load().psc_states_download(st.ptr, q.ctypes.data, depth.ctypes.data, stack.ctypes.data,
                                      status.ctypes.data, _stream(stream)))
    return {"q": q, "depth": depth, "stack": stack, "status": status}


def psc_fill_apply_noalloc(h: Handle, q, depth, status, stack, logits, bitmask_out=None, V: int | None = None,
                           stream=None):
    """psc_fill_apply on caller-owned state arrays (q, depth, status int32 [B];
    stack uint16 [B][cap] as a torch int16/uint16 tensor); allocates nothing."""
    import torch
    B = q.numel()
    V = h.V if V is None else V
    if stack.dim() != 2 or stack.shape[0] != B or not stack.is_contiguous() or stack.element_size() != 2:
        raise ValueError("stack must be a contiguous [B, cap] 16-bit tensor")
    if logits.dim() != 2 or logits.shape[0] != B or logits.shape[1] < V:
        raise ValueError("logits must be [B, >=V]")
    if bitmask_out is not None and (bitmask_out.shape != (B, h.W) or not bitmask_out.is_contiguous()):
        raise ValueError(f"bitmask_out must be a contiguous [{B}, {h.W}] tensor")
    _check(load().psc_fill_apply_noalloc(h.ptr, _ptr(q, torch.int32, "q", B), _ptr(depth, torch.int32, "depth", B),
                                         _ptr(status, torch.int32, "status", B), _ptr(stack, None, "stack"),
                                         stack.shape[1], B, _ptr(logits, None, "logits"), _dtype_code(logits),
                                         _row_stride(logits), V, _ptr(bitmask_out, torch.int32, "bitmask_out"),
                                         _stream(stream)))
