"""The allocation-free learn entry point against the store-based one.

f2_learn_batched_noalloc serves callers that cannot call cudaMalloc (device
memory pre-reserved by a pooling allocator, or code that must avoid the
implicit synchronization of cudaMalloc/cudaFree): it keeps its scheduling
scratch in a fixed device array of the library and writes the learned state
into buffers the caller owns.  Two incremental calls in a row must leave the
caller's state bit-identical to what f2_learn_batched leaves in a store after
the same two calls, and a call after the first must not change the device's
free memory.  This file is collected last on purpose.
"""
import numpy as np
import pytest

from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, csr_from_rows, cuda_device, dev_arrays, lib

pytestmark = pytest.mark.gpu


def _two_batches(wl):
    """Split every context's stream into two incremental CSR batches."""
    C = wl.num_ctx
    Wc = (wl.n_bits.astype(np.int64) + 31) // 32
    out = []
    for part in range(2):
        lo = wl.row_off[:-1] + (wl.rows * part) // 2
        hi = wl.row_off[:-1] + (wl.rows * (part + 1)) // 2
        cnt = hi - lo
        ro = np.zeros(C + 1, np.int64)
        ro[1:] = np.cumsum(cnt)
        xs = np.concatenate([wl.x[wl.x_off[c] + (lo[c] - wl.row_off[c]) * Wc[c]:
                                  wl.x_off[c] + (hi[c] - wl.row_off[c]) * Wc[c]] for c in range(C)])
        xo = np.zeros(C, np.int64)
        xo[1:] = np.cumsum(cnt * Wc)[:-1]
        ys = np.concatenate([wl.y[lo[c]:hi[c]] for c in range(C)])
        out.append((ro, xo, xs, ys))
    return out


def _caller_state(store, dev):
    """Caller-owned state buffers in the canonical layout, initialised as the
    header requires (zero, first_contra = -1)."""
    import torch

    C = store.num_ctx
    st = {
        "rank": torch.zeros(C, dtype=torch.int32, device=dev),
        "pivot_mask": torch.zeros(int(store.pw_off[-1]), dtype=torch.int32, device=dev),
        "basis_x": torch.zeros(int(store.xw_off[-1]), dtype=torch.int32, device=dev),
        "basis_z": torch.zeros((int(store.slot_off[-1]), 4), dtype=torch.int32, device=dev),
        "contra": torch.zeros(C, dtype=torch.uint8, device=dev),
        "first_contra": torch.full((C,), -1, dtype=torch.int64, device=dev),
        "n_contra": torch.zeros(C, dtype=torch.int64, device=dev),
        "rows_seen": torch.zeros(C, dtype=torch.int64, device=dev),
    }
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    return st, status


def _noalloc_call(binding, n_bits, state, status, ro, x, xo, y, raw=False):
    import torch

    nb = np.ascontiguousarray(n_bits, np.int32)
    rc = binding.load_library().f2_learn_batched_noalloc(
        int(nb.shape[0]), nb.ctypes.data, binding.F2_FLAG_RAW_FEATURES if raw else 0,
        *(state[k].data_ptr() for k in KEYS), status.data_ptr(),
        ro.data_ptr(), x.data_ptr(), xo.data_ptr(), y.data_ptr(), int(y.numel() // 4), int(x.numel()),
        int(torch.cuda.current_stream().cuda_stream))
    return rc


def _compare(binding, store, state):
    got = store.basis()
    for k in KEYS:
        a = as_bytes(binding.to_numpy(got[k]))
        b = as_bytes(binding.to_numpy(state[k]))
        assert np.array_equal(a, b), k


def _workload(kind):
    if kind in ("narrow", "raw"):
        return wlmod.generate(wlmod.scaled(2, 300), 8080)
    return wlmod.generate(dict(num_ctx=5, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=700, rows_fixed=1600,
                               dup_frac=0.0, density=0.5, n_contra=2), 8081)


@pytest.mark.parametrize("kind", ["narrow", "wide", "raw"])
def test_noalloc_matches_store_on_two_calls(kind):
    """Two calls in a row against a store: affine rows of narrow (n <= 128)
    and wide (n = 700) contexts, and raw feature rows (no constant bit)."""
    import torch

    binding = lib()
    dev = cuda_device()
    wl = _workload(kind)
    raw = kind == "raw"
    store = binding.Store(wl.n_bits, raw=raw, device=dev)
    state, status = _caller_state(store, dev)
    for ro, xo, xs, ys in _two_batches(wl):
        ro_t, xo_t, x_t, y_t = dev_arrays(binding, dev, ro, xo, xs, ys)
        store.learn(ro_t, x_t, xo_t, y_t)
        assert _noalloc_call(binding, wl.n_bits, state, status, ro_t, x_t, xo_t, y_t, raw=raw) == binding.F2_OK
        torch.cuda.synchronize()
        assert int(status.item()) == binding.F2_OK
        _compare(binding, store, state)
    assert store.device_status() == binding.F2_OK


def test_noalloc_call_allocates_nothing():
    """After the first call on the device (its one-time set-up), a call
    leaves the device's free memory and torch's allocations unchanged."""
    import torch

    binding = lib()
    dev = cuda_device()
    wl = _workload("narrow")
    store = binding.Store(wl.n_bits, device=dev)
    state, status = _caller_state(store, dev)
    batches = [dev_arrays(binding, dev, ro, xo, xs, ys) for ro, xo, xs, ys in _two_batches(wl)]
    (ro0, xo0, x0, y0), (ro1, xo1, x1, y1) = batches
    assert _noalloc_call(binding, wl.n_bits, state, status, ro0, x0, xo0, y0) == binding.F2_OK
    torch.cuda.synchronize()
    free0, used0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated(dev)
    assert _noalloc_call(binding, wl.n_bits, state, status, ro1, x1, xo1, y1) == binding.F2_OK
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert torch.cuda.memory_allocated(dev) == used0
    assert int(status.item()) == binding.F2_OK


def test_noalloc_contradiction_with_repeats():
    """A contradicting observation that is repeated: every copy counts
    (Sec. 2.2 steps (2)-(3) on each row), the first index is the first
    copy's.  The store path classifies the repeats through its duplicate
    pass, this path eliminates every row: both must give index 3, count 3."""
    import torch

    binding = lib()
    dev = cuda_device()
    n = 8
    A = [0x11, 0x23, 0x47, 0x80, 0x05, 0x0A, 0x31, 0x62]  # word bit 0 of column j (planted map)
    b = 0x9

    def word(xv, flip=0):
        w = b
        for j in range(n):
            if (xv >> j) & 1:
                w ^= A[j]
        return (np.array([w, 0, 0, 0], np.uint32) ^ np.array([flip, 0, 0, 0], np.uint32))

    # phi(7) = phi(1) + phi(2) + phi(4) (the constant bit appears three
    # times), so x = 7 lies in the span after row 2 and a flipped word there
    # is a contradiction
    rows = [(1, 0), (2, 0), (4, 0), (7, 1), (7, 1), (8, 0), (7, 1), (1, 0), (0x81, 0)]
    per_ctx = [[(np.array([xv], np.uint32), word(xv, fl)) for xv, fl in rows]]
    ro, xo, xs, ys = csr_from_rows([n], per_ctx)
    store = binding.Store(np.array([n], np.int32), device=dev)
    state, status = _caller_state(store, dev)
    ro_t, xo_t, x_t, y_t = dev_arrays(binding, dev, ro, xo, xs, ys)
    store.learn(ro_t, x_t, xo_t, y_t)
    assert _noalloc_call(binding, [n], state, status, ro_t, x_t, xo_t, y_t) == binding.F2_OK
    torch.cuda.synchronize()
    _compare(binding, store, state)
    assert int(state["contra"][0].item()) == 1
    assert int(state["first_contra"][0].item()) == 3
    assert int(state["n_contra"][0].item()) == 3


def test_noalloc_empty_call_sets_status():
    import torch

    binding = lib()
    dev = cuda_device()
    status = torch.full((1,), 7, dtype=torch.int32, device=dev)
    rc = binding.load_library().f2_learn_batched_noalloc(
        0, None, 0, *([None] * 8), status.data_ptr(), *([None] * 4), 0, 0,
        int(torch.cuda.current_stream().cuda_stream))
    assert rc == binding.F2_OK
    torch.cuda.synchronize()
    assert int(status.item()) == binding.F2_OK


def test_noalloc_rejects_oversize_and_bad_widths():
    binding = lib()
    cuda_device()
    f = binding.load_library().f2_learn_batched_noalloc
    too_many = np.ones(16385, np.int32)
    args = [None] * 9 + [None] * 4 + [0, 0, None]
    assert f(16385, too_many.ctypes.data, 0, *args) == binding.F2_ERR_INVALID_ARG
    # rejected on the host before anything is enqueued: the (host) buffer
    # below only has to look like aligned memory, it is never dereferenced
    bad = np.array([0], np.int32)
    buf = np.zeros(64, np.int64)
    p = buf.ctypes.data
    assert p % 16 == 0
    assert f(1, bad.ctypes.data, 0, *([p] * 9), *([p] * 4), 0, 0, None) == binding.F2_ERR_NBITS
