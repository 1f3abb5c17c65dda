"""Helpers shared by the GPU parity tests (CUDA path vs CPU oracle)."""
import numpy as np
import pytest

import oracle

KEYS = ("rank", "pivot_mask", "basis_x", "basis_z", "contra", "first_contra", "n_contra", "rows_seen")


def cuda_device():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.device("cuda", 0)


def lib():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2608_20532_gb300 import binding

    return binding


def dev_arrays(binding, dev, *arrays):
    return [binding.to_device(a, dev) for a in arrays]


def gpu_learn_workload(binding, store, wl, dev):
    import torch

    x_t, y_t = dev_arrays(binding, dev, wl.x, wl.y)
    for ro, xo in wl.batches:
        ro_t, xo_t = dev_arrays(binding, dev, ro, xo)
        store.learn(ro_t, x_t, xo_t, y_t)
    torch.cuda.synchronize()


def oracle_for(wl, raw=False, ctx_subset=None, threads=None):
    O = oracle.Oracle(wl.n_bits, raw=raw, threads=threads)
    for ro, xo in wl.batches:
        if ctx_subset is None:
            O.learn(ro, xo, wl.x, wl.y)
        else:
            for c in ctx_subset:
                O.learn(ro, xo, wl.x, wl.y, ctx_range=(int(c), int(c) + 1))
    return O


def as_bytes(a):
    return np.ascontiguousarray(a).reshape(-1).view(np.uint8)


def assert_basis_equal(binding, got, ref, ctx_subset=None, layout=None):
    """Bit-exact comparison of every exported array (optionally for a subset
    of contexts, using the canonical layout offsets)."""
    g = {k: binding.to_numpy(got[k]) for k in KEYS}
    if ctx_subset is None:
        for k in KEYS:
            a, b = as_bytes(g[k]), as_bytes(ref[k])
            if not np.array_equal(a, b):
                bad = np.flatnonzero(a != b)[:8]
                raise AssertionError(f"{k} differs at bytes {bad.tolist()}")
        return
    L = layout
    for c in ctx_subset:
        c = int(c)
        for k in ("rank", "contra", "first_contra", "n_contra", "rows_seen"):
            assert as_bytes(g[k][c:c + 1]).tobytes() == as_bytes(ref[k][c:c + 1]).tobytes(), (k, c)
        sl = slice(int(L["pw_off"][c]), int(L["pw_off"][c + 1]))
        assert np.array_equal(as_bytes(g["pivot_mask"][sl]), as_bytes(ref["pivot_mask"][sl])), ("pivot", c)
        sl = slice(int(L["xw_off"][c]), int(L["xw_off"][c + 1]))
        assert np.array_equal(as_bytes(g["basis_x"][sl]), as_bytes(ref["basis_x"][sl])), ("basis_x", c)
        sl = slice(int(L["slot_off"][c]), int(L["slot_off"][c + 1]))
        assert np.array_equal(as_bytes(g["basis_z"][sl]), as_bytes(ref["basis_z"][sl])), ("basis_z", c)


def csr_from_rows(n_bits, rows_per_ctx):
    """Build a CSR batch from per-context lists of (x_words[np.uint32], y_words)."""
    C = len(n_bits)
    cnt = np.array([len(r) for r in rows_per_ctx], np.int64)
    row_off = np.zeros(C + 1, np.int64)
    row_off[1:] = np.cumsum(cnt)
    W = (np.asarray(n_bits, np.int64) + 31) // 32
    x_off = np.zeros(C, np.int64)
    x_off[1:] = np.cumsum(cnt * W)[:-1]
    x = np.zeros(int((cnt * W).sum()) or 1, np.uint32)
    y = np.zeros((int(cnt.sum()) or 1, 4), np.uint32)
    for c, rows in enumerate(rows_per_ctx):
        for i, (xw, yw) in enumerate(rows):
            x[x_off[c] + i * W[c]: x_off[c] + (i + 1) * W[c]] = xw
            y[row_off[c] + i] = yw
    return row_off, x_off, x, y


def oracle_for_contexts(wl, ctxs, threads=None):
    """Oracle over the rows of the chosen contexts only (all batches, stream
    order), learned in parallel.  Returns (oracle, export); context ctxs[j]
    is the oracle's context j."""
    ctxs = np.asarray(ctxs)
    xs, ys, rows = [], [], []
    for c in ctxs:
        x, y = wl.ctx_rows(int(c))
        xs.append(np.ascontiguousarray(x).reshape(-1))
        ys.append(np.ascontiguousarray(y))
        rows.append(len(y))
    nb = wl.n_bits[ctxs]
    W = (nb.astype(np.int64) + 31) // 32
    cnt = np.array(rows, np.int64)
    row_off = np.zeros(len(ctxs) + 1, np.int64)
    row_off[1:] = np.cumsum(cnt)
    x_off = np.concatenate([[0], np.cumsum(cnt * W)[:-1]]).astype(np.int64)
    O = oracle.Oracle(nb, threads=threads or len(ctxs))
    O.learn(row_off, x_off, np.concatenate(xs), np.concatenate(ys))
    return O, O.export()


def assert_contexts_equal(binding, got, store, ref, ref_layout, ctxs):
    """Context ctxs[j] of the GPU store equals context j of the oracle."""
    g = {k: binding.to_numpy(got[k]) for k in KEYS}
    for j, c in enumerate(np.asarray(ctxs)):
        c = int(c)
        for k in ("rank", "contra", "first_contra", "n_contra", "rows_seen"):
            assert as_bytes(g[k][c:c + 1]).tobytes() == as_bytes(ref[k][j:j + 1]).tobytes(), (k, c)
        pairs = (("pivot_mask", store.pw_off, "pw_off"), ("basis_x", store.xw_off, "xw_off"),
                 ("basis_z", store.slot_off, "slot_off"))
        for k, off, lk in pairs:
            a = g[k][int(off[c]):int(off[c + 1])]
            b = ref[k][int(ref_layout[lk][j]):int(ref_layout[lk][j + 1])]
            assert np.array_equal(as_bytes(a), as_bytes(b)), (k, c)
