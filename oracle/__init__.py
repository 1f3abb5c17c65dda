"""CPU oracle for the GF(2) encoder-learning path.

TEST INFRASTRUCTURE ONLY: this package may be imported, called or executed
only by ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline /
reference arm of ``bench.py``.  The product path (the CUDA library and its
binding) never touches it, and it shares no code with that path.

Two independent restatements of the method of "Learning Exact NVIDIA SASS
Encoders with F2 Linear Algebra":

* ``f2_oracle.c`` -- plain C, one observation at a time, uint64 bitsets
  (Sec. 2.2 streaming elimination steps (1)-(5), Sec. 2.3 solve and encode);
  compiled here into ``liboracle.so`` with the host C compiler and driven
  through ctypes.  Contexts are independent, so ``Oracle.learn`` runs context
  ranges on a thread pool; nothing inside a context is reordered.
* ``f2_bigint.py`` -- Python integers, for tiny inputs and worked examples.

Every function is pinned by the ``-m "not gpu"`` tests against the paper's
worked examples (Appendices B, C, D), brute-force enumeration, planted maps
and the consistency criterion rank([Phi|Y]) = rank(Phi) (Sec. 2.3).
"""
from __future__ import annotations

import concurrent.futures as cf
import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np

from . import f2_bigint  # noqa: F401  (re-exported)

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "f2_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile f2_oracle.c into liboracle.so beside it."""
    with _lock:
        if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
            tmp = _LIB + f".{os.getpid()}.tmp"
            subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp])
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        lib.f2o_create.argtypes = [ctypes.c_int32, P, ctypes.c_int32]
        lib.f2o_create.restype = P
        lib.f2o_destroy.argtypes = [P]
        lib.f2o_destroy.restype = None
        lib.f2o_learn.argtypes = [P, ctypes.c_int32, ctypes.c_int32, P, P, P, P]
        lib.f2o_learn.restype = ctypes.c_int
        lib.f2o_export.argtypes = [P] * 9
        lib.f2o_export.restype = ctypes.c_int
        lib.f2o_solve.argtypes = [P, P]
        lib.f2o_solve.restype = ctypes.c_int
        lib.f2o_encode.argtypes = [P, ctypes.c_int64, ctypes.c_int64, P, P, ctypes.c_int32, P, P]
        lib.f2o_encode.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"], "arrays passed to the oracle must be contiguous"
    return a.ctypes.data


def layout(n_bits: np.ndarray, raw: bool = False) -> dict:
    """Offsets of the canonical exchange layout (see f2o_export)."""
    n = n_bits.astype(np.int64)
    d = n if raw else n + 1
    Wd = (d + 31) // 32
    C = n.shape[0]
    out = {"d": d, "Wd": Wd}
    for name, per in (("slot_off", d), ("xw_off", d * Wd), ("pw_off", Wd)):
        off = np.zeros(C + 1, np.int64)
        np.cumsum(per, out=off[1:])
        out[name] = off
    return out


class Oracle:
    """Per-context learning state (one plain sequential elimination per context)."""

    def __init__(self, n_bits, raw: bool = False, threads: Optional[int] = None):
        self._lib = _load()
        self.n_bits = np.ascontiguousarray(np.asarray(n_bits, np.int32))
        self.raw = bool(raw)
        self.threads = threads or max(1, os.cpu_count() or 1)
        h = self._lib.f2o_create(int(self.n_bits.shape[0]), _ptr(self.n_bits), int(self.raw))
        if not h:
            raise ValueError("oracle: feature width outside [1, 1024]")
        self._h = h
        self.layout = layout(self.n_bits, self.raw)

    def close(self):
        if getattr(self, "_h", None):
            self._lib.f2o_destroy(self._h)
            self._h = None

    def __del__(self):
        self.close()

    @property
    def num_ctx(self) -> int:
        return int(self.n_bits.shape[0])

    def learn(self, row_off, x_off, x, y, ctx_range=None):
        """Stream one CSR batch (see f2o_learn) through every context (or ctx_range)."""
        row_off = np.ascontiguousarray(row_off, np.int64)
        x_off = np.ascontiguousarray(x_off, np.int64)
        x = np.ascontiguousarray(x, np.uint32)
        y = np.ascontiguousarray(y, np.uint32)
        c0, c1 = ctx_range if ctx_range is not None else (0, self.num_ctx)
        if c1 <= c0:
            return
        d = self.layout["d"]
        work = (row_off[c0 + 1:c1 + 1] - row_off[c0:c1]).astype(np.float64) * (d[c0:c1] + 64)
        total = float(work.sum())
        target = max(total / (self.threads * 16), 1.0)
        chunks, start, acc = [], c0, 0.0
        for i, wv in enumerate(work):
            acc += wv
            if acc >= target:
                chunks.append((start, c0 + i + 1))
                start, acc = c0 + i + 1, 0.0
        if start < c1:
            chunks.append((start, c1))
        args = (_ptr(row_off), _ptr(x_off), _ptr(x), _ptr(y))

        def run(ch):
            rc = self._lib.f2o_learn(self._h, ch[0], ch[1], *args)
            if rc != 0:
                raise ValueError("oracle: invalid CSR batch")

        if self.threads == 1 or len(chunks) == 1:
            for ch in chunks:
                run(ch)
        else:
            with cf.ThreadPoolExecutor(self.threads) as ex:
                list(ex.map(run, chunks))

    def learn_workload(self, wl):
        for ro, xo in wl.batches:
            self.learn(ro, xo, wl.x, wl.y)

    def export(self) -> dict:
        L = self.layout
        C = self.num_ctx
        out = {
            "rank": np.zeros(C, np.int32),
            "pivot_mask": np.zeros(int(L["pw_off"][-1]), np.uint32),
            "basis_x": np.zeros(int(L["xw_off"][-1]), np.uint32),
            "basis_z": np.zeros((int(L["slot_off"][-1]), 4), np.uint32),
            "contra": np.zeros(C, np.uint8),
            "first_contra": np.zeros(C, np.int64),
            "n_contra": np.zeros(C, np.uint64),
            "rows_seen": np.zeros(C, np.int64),
        }
        self._lib.f2o_export(self._h, *(_ptr(out[k]) for k in (
            "rank", "pivot_mask", "basis_x", "basis_z", "contra", "first_contra", "n_contra",
            "rows_seen")))
        return out

    def solve(self) -> np.ndarray:
        W = np.zeros((int(self.layout["slot_off"][-1]), 4), np.uint32)
        self._lib.f2o_solve(self._h, _ptr(W))
        return W

    def encode(self, ctx_id, x, x_stride: Optional[int] = None):
        ctx_id = np.ascontiguousarray(ctx_id, np.int32)
        x = np.ascontiguousarray(x, np.uint32)
        Q = int(ctx_id.shape[0])
        stride = int(x_stride if x_stride is not None else (x.shape[1] if x.ndim == 2 else 1))
        y = np.zeros((Q, 4), np.uint32)
        ok = np.zeros(Q, np.uint8)
        if Q == 0:
            return y, ok
        nchunk = max(1, min(self.threads * 4, Q // 4096 + 1))
        bounds = np.linspace(0, Q, nchunk + 1).astype(np.int64)
        args = (_ptr(ctx_id), _ptr(x), stride, _ptr(y), _ptr(ok))

        def run(i):
            self._lib.f2o_encode(self._h, int(bounds[i]), int(bounds[i + 1]), *args)

        if self.threads == 1 or nchunk == 1:
            for i in range(nchunk):
                run(i)
        else:
            with cf.ThreadPoolExecutor(self.threads) as ex:
                list(ex.map(run, range(nchunk)))
        return y, ok


def ctx_view(export: dict, lay: dict, c: int) -> dict:
    """Context c's slice of an exported basis (canonical layout)."""
    d = int(lay["d"][c])
    Wd = int(lay["Wd"][c])
    s0 = int(lay["slot_off"][c])
    x0 = int(lay["xw_off"][c])
    p0 = int(lay["pw_off"][c])
    return {
        "d": d,
        "Wd": Wd,
        "rank": int(export["rank"][c]),
        "pivot_mask": export["pivot_mask"][p0:p0 + Wd],
        "basis_x": export["basis_x"][x0:x0 + d * Wd].reshape(d, Wd),
        "basis_z": export["basis_z"][s0:s0 + d],
        "contra": int(export["contra"][c]),
        "first_contra": int(export["first_contra"][c]),
        "n_contra": int(export["n_contra"][c]),
        "rows_seen": int(export["rows_seen"][c]),
    }
