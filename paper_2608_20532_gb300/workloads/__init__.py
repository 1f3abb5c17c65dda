"""Seeded synthetic workloads for the GF(2) encoder-learning path.

Input synthesis only (planted affine maps, field-structured features,
duplicates, injected contradictions, span-structured queries); it holds no
elimination, solve or encode arithmetic.  Both the CPU oracle and the CUDA path
consume the arrays built here.  The bulk work is done by ``f2gen.c`` (compiled
on first use with the host C compiler into ``libf2gen.so`` beside it).

Workloads stand in for the paper's instruction corpora (Sec. 3, Sec. 4.2:
77,926 exact contexts of joint Blackwell training), which are not available;
see the configuration table ``CONFIGS``.

Layout of a ``Workload`` (every array is a numpy array):

* ``n_bits[c]``      feature bits n_c of context c (d_c = n_c + 1 with the constant)
* ``rows[c]``        observations of context c
* ``row_off[C+1]``   CSR offsets into ``y`` (rows of c are contiguous, stream order)
* ``x_off[C]``       word offset of context c's first row in ``x``;
                     row i of c has W_c = ceil(n_c/32) words at x_off[c] + i*W_c
* ``x``              uint32 feature words, bits >= n_c zero
* ``y``              uint32[R, 4] 128-bit words (bit i = bit i%32 of word i/32)
* ``A``/``a_off``/``b``  planted map: column j of context c is A[a_off[c] + j]
* ``contra_pos[c]``  stream index (within c) of the injected contradiction, -1 if none
* ``batches``        list of (row_off, x_off) CSR views, one per incremental call
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "f2gen.c")
_LIB = os.path.join(_HERE, "libf2gen.so")
_lock = threading.Lock()
_lib = None

LAYOUT_REGS_IMM16_ONEHOT = 0
LAYOUT_CYCLIC_FIELDS = 1
LAYOUT_UNIFORM_BITS = 2


class _Params(ctypes.Structure):
    _fields_ = [
        ("num_ctx", ctypes.c_int32),
        ("layout", ctypes.c_int32),
        ("n_fixed", ctypes.c_int32),
        ("n_min", ctypes.c_int32),
        ("n_max", ctypes.c_int32),
        ("pad0", ctypes.c_int32),
        ("n_median", ctypes.c_double),
        ("n_sigma", ctypes.c_double),
        ("rows_fixed", ctypes.c_int64),
        ("rows_median", ctypes.c_double),
        ("rows_sigma", ctypes.c_double),
        ("rows_max", ctypes.c_int64),
        ("dup_frac", ctypes.c_double),
        ("density", ctypes.c_double),
        ("n_contra", ctypes.c_int32),
        ("n_two_stream", ctypes.c_int32),
        ("batch_rows", ctypes.c_int64),
    ]


def build_generator(force: bool = False) -> str:
    """Compile f2gen.c into libf2gen.so beside it (host C compiler)."""
    with _lock:
        if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
            tmp = _LIB + f".{os.getpid()}.tmp"
            subprocess.check_call(
                ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", _SRC, "-o", tmp, "-lm"])
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build_generator())
        P = ctypes.c_void_p
        lib.f2gen_plan.argtypes = [ctypes.POINTER(_Params), ctypes.c_uint64, P, P, P, P, P]
        lib.f2gen_plan.restype = ctypes.c_int
        lib.f2gen_fill.argtypes = [ctypes.POINTER(_Params), ctypes.c_uint64] + [P] * 14 + [ctypes.c_int32]
        lib.f2gen_fill.restype = ctypes.c_int
        lib.f2gen_queries.argtypes = [
            ctypes.c_uint64, ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, P, P, P, P, P, P,
            ctypes.c_int32, ctypes.c_double, ctypes.c_int64, ctypes.c_double, ctypes.c_int32, P, P, P,
            ctypes.c_int32]
        lib.f2gen_queries.restype = ctypes.c_int
        lib.f2gen_onehot_offset.argtypes = [ctypes.c_int32]
        lib.f2gen_onehot_offset.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def _threads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


# Configurations (seeded 20260000 + k).  Readings of unstated details:
# counts "x% of contexts" are round(x*C) (at least 1); duplicate rows copy
# earlier fresh rows; an injected contradiction is a duplicate observation
# with one flipped y bit (guaranteed in the span of earlier rows).
CONFIGS = {
    # 256 contexts, n = 48 (three 8-bit registers, a 16-bit immediate, 8
    # one-hot modifier bits), A 128x48 at density 0.1, 200 observations + 30%
    # duplicates, 1% (3) contexts with a contradiction, 100 held-out queries
    # per context, half of them outside the span.
    1: dict(num_ctx=256, layout=LAYOUT_REGS_IMM16_ONEHOT, n_fixed=48, rows_fixed=200, dup_frac=0.3,
            density=0.1, n_contra=3,
            queries=dict(ctx_mode=0, per_ctx=100, out_frac=0.5)),
    # 4,096 contexts, n uniform in [32, 128], structured fields, A at density
    # 0.05, rows log-normal (median 300, max 20k), 50% duplicates, 0.5% (20)
    # contexts with a contradiction.
    2: dict(num_ctx=4096, layout=LAYOUT_CYCLIC_FIELDS, n_min=32, n_max=128, rows_median=300,
            rows_sigma=1.2, rows_max=20000, dup_frac=0.5, density=0.05, n_contra=20),
    # 77,926 contexts (joint Blackwell scale), n log-normal median 64 in
    # [16, 256], rows log-normal (median 500, max 200k, ~80M total), 85%
    # duplicates, 49,566 two-variant-stream contexts, no contradictions.
    3: dict(num_ctx=77926, layout=LAYOUT_CYCLIC_FIELDS, n_min=16, n_max=256, n_median=64, n_sigma=0.6,
            rows_median=500, rows_sigma=1.2, rows_max=200000, dup_frac=0.85, density=0.05,
            n_contra=0, n_two_stream=49566,
            # 10M encode queries over the learned config-3 store, Zipf(1.1)
            # context ids, 5% outside the span.
            queries=dict(ctx_mode=1, count=10_000_000, zipf_s=1.1, out_frac=0.05)),
    # 64 contexts, n = 1024, dense planted A (density 0.5), 2^20 uniform rows
    # per context streamed in 16 batches of 65,536 rows, 8 contexts with a
    # contradiction in a random batch.
    5: dict(num_ctx=64, layout=LAYOUT_UNIFORM_BITS, n_fixed=1024, rows_fixed=1 << 20, dup_frac=0.0,
            density=0.5, n_contra=8, batch_rows=65536),
}


def seed_for(cfg_id: int) -> int:
    return 20260000 + cfg_id


@dataclasses.dataclass
class Queries:
    ctx_id: np.ndarray      # int32[Q]
    x: np.ndarray           # uint32[Q, stride]
    stride: int
    expect_in: np.ndarray   # uint8[Q], 1 = in-span construction


@dataclasses.dataclass
class Workload:
    name: str
    params: dict
    seed: int
    n_bits: np.ndarray
    rows: np.ndarray
    fresh: np.ndarray
    dups: np.ndarray
    contra: np.ndarray
    two_stream: np.ndarray
    row_off: np.ndarray
    x_off: np.ndarray
    x: np.ndarray
    y: np.ndarray
    a_off: np.ndarray
    A: np.ndarray
    b: np.ndarray
    contra_pos: np.ndarray
    contra_bit: np.ndarray
    batches: list
    queries: Optional[Queries] = None

    @property
    def num_ctx(self) -> int:
        return int(self.n_bits.shape[0])

    @property
    def total_rows(self) -> int:
        return int(self.rows.sum())

    def words(self) -> np.ndarray:
        return (self.n_bits.astype(np.int64) + 31) // 32

    def ctx_rows(self, c: int):
        """(x[T, W], y[T, 4]) of context c in stream order (copies for batch-major data)."""
        W = int((self.n_bits[c] + 31) // 32)
        T = int(self.rows[c])
        if len(self.batches) == 1:
            r0 = int(self.row_off[c])
            x0 = int(self.x_off[c])
            return (self.x[x0:x0 + T * W].reshape(T, W), self.y[r0:r0 + T])
        xs, ys = [], []
        for ro, xo in self.batches:
            t = int(ro[c + 1] - ro[c])
            xs.append(self.x[int(xo[c]):int(xo[c]) + t * W].reshape(t, W))
            ys.append(self.y[int(ro[c]):int(ro[c]) + t])
        return np.concatenate(xs), np.concatenate(ys)

    def algorithmic_bytes(self) -> int:
        """Bytes a learn pass must read: packed x (ceil(n/8) B) + 16 B of y per row."""
        return int((self.rows * ((self.n_bits.astype(np.int64) + 7) // 8 + 16)).sum())


def _params(cfg: dict) -> _Params:
    p = _Params()
    p.num_ctx = cfg["num_ctx"]
    p.layout = cfg["layout"]
    p.n_fixed = cfg.get("n_fixed", 0)
    p.n_min = cfg.get("n_min", 1)
    p.n_max = cfg.get("n_max", 1024)
    p.n_median = cfg.get("n_median", 0.0)
    p.n_sigma = cfg.get("n_sigma", 0.0)
    p.rows_fixed = cfg.get("rows_fixed", 0)
    p.rows_median = cfg.get("rows_median", 1.0)
    p.rows_sigma = cfg.get("rows_sigma", 0.0)
    p.rows_max = cfg.get("rows_max", 1)
    p.dup_frac = cfg.get("dup_frac", 0.0)
    p.density = cfg.get("density", 0.5)
    p.n_contra = cfg.get("n_contra", 0)
    p.n_two_stream = cfg.get("n_two_stream", 0)
    p.batch_rows = cfg.get("batch_rows", 0)
    return p


def config(cfg_id: int, **overrides) -> dict:
    """A copy of configuration cfg_id with overrides applied."""
    cfg = dict(CONFIGS[cfg_id])
    cfg.update(overrides)
    return cfg


def scaled(cfg_id: int, num_ctx: int, **overrides) -> dict:
    """Configuration cfg_id with fewer contexts; contradiction and two-stream
    counts shrink in proportion (at least one contradiction context if the
    full configuration has any)."""
    base = CONFIGS[cfg_id]
    f = num_ctx / base["num_ctx"]
    cfg = dict(base)
    cfg["num_ctx"] = num_ctx
    if base.get("n_contra", 0):
        cfg["n_contra"] = max(1, int(round(base["n_contra"] * f)))
    if base.get("n_two_stream", 0):
        cfg["n_two_stream"] = int(round(base["n_two_stream"] * f))
    cfg.update(overrides)
    return cfg


def generate(cfg: dict, seed: int, name: str = "custom", nthreads: Optional[int] = None,
             query_count: Optional[int] = None) -> Workload:
    """Build the workload described by cfg (see CONFIGS) with the given seed."""
    lib = _load()
    p = _params(cfg)
    C = p.num_ctx
    n_bits = np.zeros(C, np.int32)
    fresh = np.zeros(C, np.int64)
    dups = np.zeros(C, np.int64)
    contra = np.zeros(C, np.uint8)
    two = np.zeros(C, np.uint8)
    if lib.f2gen_plan(ctypes.byref(p), seed, _ptr(n_bits), _ptr(fresh), _ptr(dups), _ptr(contra),
                      _ptr(two)) != 0:
        raise ValueError("invalid workload parameters")
    rows = fresh + dups
    W = (n_bits.astype(np.int64) + 31) // 32
    R = int(rows.sum())
    batch_rows = int(cfg.get("batch_rows", 0))
    if batch_rows:
        if len(set(rows.tolist())) != 1 or len(set(n_bits.tolist())) != 1 or rows[0] % batch_rows:
            raise ValueError("batch-major layout needs equal rows (a multiple of batch_rows) and n")
        nb = int(rows[0]) // batch_rows
        w = int(W[0])
        batches = []
        for bi in range(nb):
            ro = (bi * C * batch_rows + np.arange(C + 1, dtype=np.int64) * batch_rows)
            batches.append((ro, ro[:-1] * w))
        row_off = batches[0][0]
        x_off = batches[0][1]
    else:
        row_off = np.zeros(C + 1, np.int64)
        np.cumsum(rows, out=row_off[1:])
        x_off = np.zeros(C, np.int64)
        np.cumsum((rows * W)[:-1], out=x_off[1:])
        batches = [(row_off, x_off)]
    x = np.zeros(int((rows * W).sum()), np.uint32)
    y = np.zeros((R, 4), np.uint32)
    a_off = np.zeros(C, np.int64)
    np.cumsum(n_bits[:-1].astype(np.int64), out=a_off[1:])
    A = np.zeros((int(n_bits.astype(np.int64).sum()), 4), np.uint32)
    b = np.zeros((C, 4), np.uint32)
    contra_pos = np.full(C, -1, np.int64)
    contra_bit = np.full(C, -1, np.int32)
    nt = nthreads or _threads()
    if lib.f2gen_fill(ctypes.byref(p), seed, _ptr(n_bits), _ptr(fresh), _ptr(dups), _ptr(contra),
                      _ptr(two), _ptr(row_off), _ptr(x_off), _ptr(x), _ptr(y), _ptr(A), _ptr(a_off),
                      _ptr(b), _ptr(contra_pos), _ptr(contra_bit), nt) != 0:
        raise MemoryError("workload fill failed")
    wl = Workload(name=name, params=dict(cfg), seed=seed, n_bits=n_bits, rows=rows, fresh=fresh,
                  dups=dups, contra=contra, two_stream=two, row_off=row_off, x_off=x_off, x=x, y=y,
                  a_off=a_off, A=A, b=b, contra_pos=contra_pos, contra_bit=contra_bit,
                  batches=batches)
    qcfg = cfg.get("queries")
    if qcfg is not None:
        wl.queries = make_queries(wl, qcfg, seed, count=query_count, nthreads=nt)
    return wl


def make_queries(wl: Workload, qcfg: dict, seed: int, count: Optional[int] = None,
                 nthreads: Optional[int] = None) -> Queries:
    """Queries over wl's training rows (CSR layout only); see f2gen_queries."""
    if len(wl.batches) != 1:
        raise ValueError("queries need a CSR (single-batch) workload")
    lib = _load()
    C = wl.num_ctx
    mode = int(qcfg["ctx_mode"])
    if mode == 0:
        per = int(qcfg["per_ctx"])
        Q = per * C if count is None else int(count)
    else:
        per = 0
        Q = int(qcfg["count"]) if count is None else int(count)
    stride = int(((wl.n_bits.astype(np.int64) + 31) // 32).max())
    ctx_id = np.zeros(Q, np.int32)
    qx = np.zeros((Q, stride), np.uint32)
    expect = np.zeros(Q, np.uint8)
    rc = lib.f2gen_queries(seed + 1_000_003, int(wl.params["layout"]), Q, C, _ptr(wl.n_bits),
                           _ptr(wl.rows), _ptr(wl.row_off), _ptr(wl.x_off), _ptr(wl.x),
                           _ptr(wl.contra_pos), mode, float(qcfg.get("zipf_s", 1.0)), per,
                           float(qcfg.get("out_frac", 0.0)), stride, _ptr(ctx_id), _ptr(qx),
                           _ptr(expect), nthreads or _threads())
    if rc != 0:
        raise ValueError("invalid query parameters")
    return Queries(ctx_id=ctx_id, x=qx, stride=stride, expect_in=expect)


def onehot_offset(layout: int) -> int:
    return int(_load().f2gen_onehot_offset(layout))


def standard(cfg_id: int, **kw) -> Workload:
    """Configuration cfg_id at full size with its standard seed."""
    return generate(CONFIGS[cfg_id], seed_for(cfg_id), name=f"config{cfg_id}", **kw)


# Parsed-value workload with the paper's exact-context rank statistics (input
# synthesis only).  A context's observations carry k parsed int64 values;
# phi(x) = [1 || bits64(v_0) || ... || bits64(v_{k-1})] (Sec. 2.1), so the
# k values of a row, little-endian, are its n = 64k feature bits: x below is
# the int64 values' memory seen as uint32 words.  Per context the evidence
# rank r (of the [1 || x] rows) is log-normal with median 3 and 95th
# percentile 21 (the SM107 statistics of Sec. 4), rows are ~200 per rank
# (the ~200x compaction of the corpora), and x = offset XOR a random subset
# of r - 1 sparse generators that flip low-order, mid-order or sign bits of
# one value (register-, immediate- and sign-like fields).  y is a planted
# affine map of x; a few contexts get one duplicate x with a flipped y bit.
# Consecutive contexts in groups of group_size share k and the planted map:
# the exact contexts of one (f, m) group, which differ in their operand
# signature (and so in their input subspace) but not in the map (Sec. 3).
PARSED_LOWRANK = dict(num_ctx=10000, k_min=2, k_max=8, rank_median=3.0, rank_p95=21.0, rows_per_rank=200,
                      rows_max=1 << 16, density=0.05, n_contra=20, group_size=8)


def parsed_lowrank(seed: int = 20260006, **over) -> Workload:
    p = dict(PARSED_LOWRANK, **over)
    rng = np.random.default_rng(seed)
    C = int(p["num_ctx"])
    gs = max(1, int(p["group_size"]))
    k = np.repeat(rng.integers(int(p["k_min"]), int(p["k_max"]) + 1, (C + gs - 1) // gs), gs)[:C]
    n_bits = (64 * k).astype(np.int32)
    sigma = np.log(p["rank_p95"] / p["rank_median"]) / 1.6449
    r = np.rint(np.exp(rng.normal(np.log(p["rank_median"]), sigma, C))).astype(np.int64)
    r = np.clip(r, 1, 64)
    T = np.rint(r * p["rows_per_rank"] * np.exp(rng.normal(0.0, 0.5, C))).astype(np.int64)
    T = np.clip(T, np.maximum(r, 2), int(p["rows_max"]))
    contra_ctx = rng.choice(C, size=min(C, int(p["n_contra"])), replace=False)
    W = (n_bits.astype(np.int64) + 31) // 32  # = 2k
    row_off = np.zeros(C + 1, np.int64)
    row_off[1:] = np.cumsum(T)
    x_off = np.zeros(C, np.int64)
    x_off[1:] = np.cumsum(T * W)[:-1]
    R = int(T.sum())
    x64 = np.zeros(int((T * k).sum()), np.int64)
    y = np.zeros((R, 4), np.uint32)
    a_off = np.zeros(C, np.int64)
    a_off[1:] = np.cumsum(n_bits.astype(np.int64))[:-1]
    A = np.zeros((int(n_bits.sum()), 4), np.uint32)
    b = np.zeros((C, 4), np.uint32)
    contra_pos = np.full(C, -1, np.int64)
    contra_bit = np.full(C, -1, np.int32)
    is_contra = np.zeros(C, bool)
    is_contra[contra_ctx] = True
    for c in range(C):
        kc, n, Tc, rc = int(k[c]), int(n_bits[c]), int(T[c]), int(r[c])
        if c % gs == 0:  # planted map of the group: column j of A is the word of feature bit j
            Ac = (rng.random((n, 128)) < p["density"])
            Aw = np.packbits(Ac, axis=1, bitorder="little").view(np.uint32).reshape(n, 4)
            bc = rng.integers(0, 2 ** 32, size=4, dtype=np.uint64).astype(np.uint32)
        A[a_off[c]:a_off[c] + n] = Aw
        b[c] = bc
        # offset values (small, sometimes negative) and sparse generators
        off = rng.integers(0, 256, kc).astype(np.int64)
        off[rng.random(kc) < 0.1] *= -1
        gens = np.zeros((max(rc - 1, 0), kc), np.int64)
        for j in range(rc - 1):
            i = rng.integers(kc)
            u = rng.random()
            bit = int(rng.integers(8)) if u < 0.6 else (int(rng.integers(8, 32)) if u < 0.95 else 63)
            gens[j, i] = np.int64(1) << np.int64(bit) if bit < 63 else np.int64(-(1 << 63))
        sel = rng.random((Tc, max(rc - 1, 0))) < 0.5
        xv = np.tile(off, (Tc, 1))
        for j in range(rc - 1):
            xv[sel[:, j]] ^= gens[j]
        # y = b XOR A x, evaluated through the generators (x is affine in sel)
        def word(vals):
            bits = np.unpackbits(vals.astype("<i8").view(np.uint8), bitorder="little")[:n].astype(bool)
            return np.bitwise_xor.reduce(Aw[bits], axis=0) if bits.any() else np.zeros(4, np.uint32)
        y_off = bc ^ word(off)
        yc = np.tile(y_off, (Tc, 1))
        for j in range(rc - 1):
            yc[sel[:, j]] ^= word(gens[j])
        if is_contra[c] and Tc > 1:
            # a later copy of an earlier row's x with one flipped word bit
            pos = int(rng.integers(1, Tc))
            src = int(rng.integers(0, pos))
            xv[pos] = xv[src]
            yc[pos] = yc[src]
            bit = int(rng.integers(128))
            yc[pos, bit // 32] ^= np.uint32(1 << (bit % 32))
            contra_pos[c] = pos
            contra_bit[c] = bit
        x64[x_off[c] // 2: x_off[c] // 2 + Tc * kc] = xv.reshape(-1)
        y[row_off[c]:row_off[c + 1]] = yc
    x = x64.view(np.uint32)
    zeros = np.zeros(C, np.int64)
    return Workload(name="parsed-lowrank", params=p, seed=seed, n_bits=n_bits, rows=T, fresh=r, dups=T - r,
                    contra=is_contra.astype(np.uint8), two_stream=np.zeros(C, np.uint8), row_off=row_off,
                    x_off=x_off, x=x, y=y, a_off=a_off, A=A, b=b, contra_pos=contra_pos, contra_bit=contra_bit,
                    batches=[(row_off, x_off)], queries=None)
