"""Thin Python binding of libf2gpu.so (argument marshalling only).

Every step of the learning path runs in the library's CUDA kernels; this
module only passes device pointers (``tensor.data_ptr()``), sizes and the
current CUDA stream through the C ABI declared in ``include/f2gpu.h``.
PyTorch provides device memory and streams.  There is no CPU fallback: if
the library is missing the first call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np
import torch

from . import build as _build

F2_OK = 0
F2_ERR_INVALID_ARG = 1
F2_ERR_NBITS = 2
F2_ERR_CTX_RANGE = 3
F2_ERR_ALIGN = 4
F2_ERR_OOM = 5
F2_ERR_CUDA = 6
F2_ERR_TIMEOUT = 7
F2_ERR_ROWS = 8
F2_ERR_STRIDE = 9
F2_FLAG_RAW_FEATURES = 1
F2_OPT_HEAVY_ROWS = 1
F2_OPT_WARP_BASIS_BYTES = 2
F2_OPT_WARP_WORK = 3
F2_OPT_DEDUP = 4
F2_OPT_ENCODE_TABLE_MIN = 5
F2_OPT_HOST_CHUNK_BYTES = 6
F2_OPT_ENCODE_CHUNK_SHIFT = 7
F2_OPT_ENCODE_CHUNK_MIN = 8
F2_OPT_FAIL_ALLOC = 9
F2_OPT_TIMING = 10
F2_OPT_ELIM_TABLES = 11
F2_OPT_SMALL_BASIS_BYTES = 12
F2_OPT_DEDUP_SHARDS = 13
F2_OPT_ENCODE_DIRECT_MAX = 14
F2_OPT_LONG_CALL_ROWS = 15
F2_OPT_HANDOFF_REPS = 16

# every entry point of include/f2gpu.h
EXPORTS = (
    "f2_status_string", "f2_create", "f2_destroy", "f2_reset", "f2_layout", "f2_sizes",
    "f2_learn_batched", "f2_get_basis", "f2_solve_affine", "f2_encode_batched", "f2_device_status",
    "f2_store_export", "f2_store_import", "f2_set_option", "f2_peak_lop3", "f2_learn_batched_noalloc",
    "f2_encode_epilogue", "f2_merge_bases", "f2_learn_host", "f2_encode_host", "f2_learn_timing",
)

_lib = None


class F2Error(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = code
        super().__init__(f"{what}: {status_string(code)} ({code})")


def library_path() -> str:
    return _build.LIB


def load_library(path: Optional[str] = None):
    """Load libf2gpu.so (built by ``__graft_entry__.build()``); raises if absent."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or library_path()
    if not os.path.exists(p):
        raise RuntimeError(f"libf2gpu.so not built ({p}); run __graft_entry__.build() first")
    lib = ctypes.CDLL(p)
    P = ctypes.c_void_p
    i32, i64, u32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    sig = {
        "f2_status_string": ([ctypes.c_int], ctypes.c_char_p),
        "f2_create": ([ctypes.POINTER(P), i32, P, u32, P], ctypes.c_int),
        "f2_destroy": ([P], None),
        "f2_reset": ([P, P], ctypes.c_int),
        "f2_layout": ([P, P, P, P], ctypes.c_int),
        "f2_sizes": ([P, P, P, P, P], ctypes.c_int),
        "f2_learn_batched": ([P, P, P, P, P, i64, i64, P], ctypes.c_int),
        "f2_get_basis": ([P] + [P] * 8 + [P], ctypes.c_int),
        "f2_solve_affine": ([P, P, P], ctypes.c_int),
        "f2_encode_batched": ([P, i64, P, P, i32, P, P, P], ctypes.c_int),
        "f2_learn_host": ([P, P, P, P, P, i64, i64, P], ctypes.c_int),
        "f2_encode_host": ([P, i64, P, P, i32, P, P, P], ctypes.c_int),
        "f2_encode_epilogue": ([P, i64, P, P, P, P, P, P, P], ctypes.c_int),
        "f2_merge_bases": ([P, i32, P, P, ctypes.POINTER(P), P, P], ctypes.c_int),
        "f2_device_status": ([P, ctypes.POINTER(ctypes.c_int), P], ctypes.c_int),
        "f2_store_export": ([P, P, ctypes.POINTER(ctypes.c_size_t), P], ctypes.c_int),
        "f2_store_import": ([P, P, ctypes.c_size_t, P], ctypes.c_int),
        "f2_set_option": ([P, ctypes.c_int, i64], ctypes.c_int),
        "f2_peak_lop3": ([P, i32, i32, ctypes.POINTER(i64), P], ctypes.c_int),
        "f2_learn_batched_noalloc": ([i32, P, u32] + [P] * 9 + [P, P, P, P, i64, i64, P], ctypes.c_int),
        "f2_learn_timing": ([P, P, P], ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    if path is None:
        _lib = lib
    return lib


def status_string(code: int) -> str:
    try:
        return load_library().f2_status_string(code).decode()
    except RuntimeError:
        return f"status {code}"


def _check(code: int, what: str):
    if code != F2_OK:
        raise F2Error(code, what)


def _stream(stream=None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _hptr(a):
    """Address of a host array (CPU tensor, ideally pinned, or numpy array)."""
    if isinstance(a, torch.Tensor):
        if a.is_cuda or not a.is_contiguous():
            raise ValueError("expected a contiguous CPU tensor")
        return a.data_ptr()
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("expected a contiguous array")
        return a.ctypes.data
    raise TypeError("expected a CPU tensor or a numpy array")


def _hsize(a) -> int:
    return a.numel() if isinstance(a, torch.Tensor) else a.size


def _dptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


class Store:
    """A set of encoding contexts and their learned reduced bases on one GPU."""

    def __init__(self, n_bits, raw: bool = False, device=None, stream=None, _handle=None):
        self._lib = load_library()
        nb = np.ascontiguousarray(np.asarray(n_bits, dtype=np.int32))
        self.n_bits = nb
        self.raw = bool(raw)
        self.device = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        if _handle is None:
            h = ctypes.c_void_p()
            with torch.cuda.device(self.device):
                _check(self._lib.f2_create(ctypes.byref(h), int(nb.shape[0]), nb.ctypes.data,
                                           F2_FLAG_RAW_FEATURES if raw else 0, _stream(stream)), "f2_create")
        else:  # a store the library created (f2_merge_bases)
            h = _handle
        self._h = h
        n = int(nb.shape[0]) + 1
        self.slot_off = np.zeros(n, np.int64)
        self.xw_off = np.zeros(n, np.int64)
        self.pw_off = np.zeros(n, np.int64)
        _check(self._lib.f2_layout(self._h, self.slot_off.ctypes.data, self.xw_off.ctypes.data,
                                   self.pw_off.ctypes.data), "f2_layout")

    def close(self):
        if getattr(self, "_h", None) and self._h.value:
            self._lib.f2_destroy(self._h)  # frees device memory: the device has synchronized
            self._h = ctypes.c_void_p()
        self._held = []

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def num_ctx(self) -> int:
        return int(self.n_bits.shape[0])

    def set_option(self, option: int, value: int):
        _check(self._lib.f2_set_option(self._h, option, int(value)), "f2_set_option")

    def reset(self, stream=None):
        _check(self._lib.f2_reset(self._h, _stream(stream)), "f2_reset")

    def learn(self, row_off: torch.Tensor, x: torch.Tensor, x_off: torch.Tensor, y: torch.Tensor, stream=None):
        """One batch: row_off int64[C+1], x int32/uint32 words, x_off int64[C], y int32[R, 4]."""
        if row_off.dtype != torch.int64 or x_off.dtype != torch.int64:
            raise TypeError("row_off and x_off must be int64")
        total_rows = y.numel() // 4
        _check(self._lib.f2_learn_batched(self._h, _dptr(row_off), _dptr(x), _dptr(x_off), _dptr(y),
                                          int(total_rows), int(x.numel()), _stream(stream)),
               "f2_learn_batched")

    def _hold(self, arrays, stream):
        """Keep host arrays alive until `stream` has passed the call that reads or writes them."""
        held = getattr(self, "_held", None)
        if held is None:
            held = self._held = []
        held[:] = [(ev, refs) for ev, refs in held if not ev.query()]
        ev = torch.cuda.Event()
        ev.record(stream if stream is not None else torch.cuda.current_stream(self.device))
        held.append((ev, tuple(arrays)))

    def learn_host(self, row_off, x, x_off, y, stream=None):
        """One batch from host memory (f2_learn_host): row_off int64[C+1], x 32-bit words,
        x_off int64[C], y 32-bit words [R, 4]; pinned CPU tensors let copies overlap."""
        with torch.cuda.device(self.device):
            _check(self._lib.f2_learn_host(self._h, _hptr(row_off), _hptr(x), _hptr(x_off), _hptr(y),
                                           int(_hsize(y) // 4), int(_hsize(x)), _stream(stream)),
                   "f2_learn_host")
            self._hold((row_off, x, x_off, y), stream)

    def encode_host(self, ctx_id, x, y_out, in_span, stream=None):
        """Queries in host memory (f2_encode_host): ctx_id int32[Q], x 32-bit words [Q, stride];
        y_out 32-bit words [Q, 4] and in_span uint8[Q] are written once `stream` passes the call."""
        Q = int(_hsize(ctx_id))
        stride = int(x.shape[1]) if len(x.shape) == 2 else 1
        with torch.cuda.device(self.device):
            _check(self._lib.f2_encode_host(self._h, Q, _hptr(ctx_id), _hptr(x), stride, _hptr(y_out),
                                            _hptr(in_span), _stream(stream)), "f2_encode_host")
            self._hold((ctx_id, x, y_out, in_span), stream)
        return y_out, in_span

    def basis(self, stream=None) -> dict:
        C = self.num_ctx
        dev = self.device
        out = {
            "rank": torch.empty(C, dtype=torch.int32, device=dev),
            "pivot_mask": torch.empty(int(self.pw_off[-1]), dtype=torch.int32, device=dev),
            "basis_x": torch.empty(int(self.xw_off[-1]), dtype=torch.int32, device=dev),
            "basis_z": torch.empty((int(self.slot_off[-1]), 4), dtype=torch.int32, device=dev),
            "contra": torch.empty(C, dtype=torch.uint8, device=dev),
            "first_contra": torch.empty(C, dtype=torch.int64, device=dev),
            "n_contra": torch.empty(C, dtype=torch.int64, device=dev),
            "rows_seen": torch.empty(C, dtype=torch.int64, device=dev),
        }
        keys = ("rank", "pivot_mask", "basis_x", "basis_z", "contra", "first_contra", "n_contra", "rows_seen")
        _check(self._lib.f2_get_basis(self._h, *(_dptr(out[k]) for k in keys), _stream(stream)), "f2_get_basis")
        return out

    def solve(self, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        if out is None:
            out = torch.empty((int(self.slot_off[-1]), 4), dtype=torch.int32, device=self.device)
        _check(self._lib.f2_solve_affine(self._h, _dptr(out), _stream(stream)), "f2_solve_affine")
        return out

    def encode(self, ctx_id: torch.Tensor, x: torch.Tensor, y_out: Optional[torch.Tensor] = None,
               in_span: Optional[torch.Tensor] = None, stream=None):
        """ctx_id int32[Q], x int32[Q, stride] -> (y int32[Q, 4], in_span uint8[Q])."""
        Q = int(ctx_id.numel())
        stride = int(x.shape[1]) if x.dim() == 2 else 1
        if y_out is None:
            y_out = torch.empty((Q, 4), dtype=torch.int32, device=self.device)
        if in_span is None:
            in_span = torch.empty(Q, dtype=torch.uint8, device=self.device)
        _check(self._lib.f2_encode_batched(self._h, Q, _dptr(ctx_id), _dptr(x), stride, _dptr(y_out),
                                           _dptr(in_span), _stream(stream)), "f2_encode_batched")
        return y_out, in_span

    def encode_epilogue(self, ctx_id: torch.Tensor, in_span: torch.Tensor, y: torch.Tensor, sched=None,
                        state=None, opaque_mask=None, stream=None):
        """Full words in place (Appendix C/D): y ^= sched << 105, then the bits
        of opaque_mask[ctx] taken from state; rejected queries untouched.
        sched int32[Q], state int32[Q, 4], opaque_mask int32[num_ctx, 4]."""
        Q = int(ctx_id.numel())
        _check(self._lib.f2_encode_epilogue(self._h, Q, _dptr(ctx_id), _dptr(in_span),
                                            _dptr(sched) if sched is not None else None,
                                            _dptr(state) if state is not None else None,
                                            _dptr(opaque_mask) if opaque_mask is not None else None,
                                            _dptr(y), _stream(stream)), "f2_encode_epilogue")
        return y

    def merge(self, group_of, num_groups: int, out_mask=None, stream=None):
        """Map pooling: the bases of each group of contexts eliminated together
        (f2_merge_bases).  Returns (store with one raw-feature context per
        group, mask_ok uint8[num_groups])."""
        g = np.ascontiguousarray(np.asarray(group_of, dtype=np.int32))
        m = None if out_mask is None else np.ascontiguousarray(np.asarray(out_mask, dtype=np.uint32))
        ok = np.zeros(max(int(num_groups), 1), np.uint8)
        h = ctypes.c_void_p()
        with torch.cuda.device(self.device):
            _check(self._lib.f2_merge_bases(self._h, int(num_groups), g.ctypes.data,
                                            m.ctypes.data if m is not None else None, ctypes.byref(h),
                                            ok.ctypes.data, _stream(stream)), "f2_merge_bases")
        d = np.zeros(int(num_groups), np.int32)
        for c in range(len(g)):
            if g[c] >= 0:
                d[g[c]] = self.n_bits[c] + (0 if self.raw else 1)
        return Store(d, raw=True, device=self.device, _handle=h), ok[:int(num_groups)]

    def learn_timing(self, stream=None) -> np.ndarray:
        """Per-context timestamps of the last learn call (F2_OPT_TIMING on):
        uint64[num_ctx, 6] = dedup start/end, elimination start/end (ns), their SM ids."""
        out = np.zeros((self.num_ctx, 6), np.uint64)
        _check(self._lib.f2_learn_timing(self._h, out.ctypes.data, _stream(stream)), "f2_learn_timing")
        return out

    def device_status(self, stream=None) -> int:
        v = ctypes.c_int(0)
        _check(self._lib.f2_device_status(self._h, ctypes.byref(v), _stream(stream)), "f2_device_status")
        return int(v.value)

    def export_state(self, stream=None) -> bytes:
        n = ctypes.c_size_t(0)
        _check(self._lib.f2_store_export(self._h, None, ctypes.byref(n), _stream(stream)), "f2_store_export")
        buf = ctypes.create_string_buffer(n.value)
        _check(self._lib.f2_store_export(self._h, buf, ctypes.byref(n), _stream(stream)), "f2_store_export")
        return buf.raw[:n.value]

    def import_state(self, data: bytes, stream=None):
        buf = ctypes.create_string_buffer(data, len(data))
        _check(self._lib.f2_store_import(self._h, buf, len(data), _stream(stream)), "f2_store_import")


def peak_lop3(blocks: int, iters: int, out: torch.Tensor, stream=None) -> int:
    """Launch the integer-pipe probe; returns the LOP3 lane-operations it executes."""
    n = ctypes.c_int64(0)
    _check(load_library().f2_peak_lop3(_dptr(out), int(blocks), int(iters), ctypes.byref(n), _stream(stream)),
           "f2_peak_lop3")
    return int(n.value)


def to_device(a: np.ndarray, device) -> torch.Tensor:
    """numpy array -> CUDA tensor (uint32 reinterpreted as int32, same bits)."""
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    elif a.dtype == np.uint64:
        a = a.view(np.int64)
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def to_numpy(t: torch.Tensor, dtype=None) -> np.ndarray:
    a = t.detach().cpu().numpy()
    if dtype is not None:
        a = a.view(dtype)
    return a
