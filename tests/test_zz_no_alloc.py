"""The allocation-free learn entry point against the store-based one.

f2_learn_batched_noalloc serves callers that cannot call cudaMalloc (device
memory pre-reserved by a pooling allocator, or code that must avoid the
implicit synchronization of cudaMalloc/cudaFree): it keeps its scheduling
scratch in a fixed device array of the library and writes the learned state
into buffers the caller owns.  Two incremental calls in a row must leave the
caller's state bit-identical to what f2_learn_batched leaves in a store after
the same two calls.  This file is collected last on purpose.
"""
import numpy as np
import pytest

from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, cuda_device, dev_arrays, lib

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


def _noalloc_call(binding, n_bits, state, status, ro, x, xo, y):
    import torch

    nb = np.ascontiguousarray(n_bits, np.int32)
    rc = binding.load_library().f2_learn_batched_noalloc(
        int(nb.shape[0]), nb.ctypes.data, 0, *(state[k].data_ptr() for k in KEYS), status.data_ptr(),
        ro.data_ptr(), x.data_ptr(), xo.data_ptr(), y.data_ptr(), int(y.numel() // 4), int(x.numel()),
        int(torch.cuda.current_stream().cuda_stream))
    return rc


def _compare(binding, store, state):
    got = store.basis()
    for k in KEYS:
        a = as_bytes(binding.to_numpy(got[k]))
        b = as_bytes(binding.to_numpy(state[k]))
        assert np.array_equal(a, b), k


@pytest.mark.parametrize("kind", ["narrow", "wide"])
def test_noalloc_matches_store_on_two_calls(kind):
    import torch

    binding = lib()
    dev = cuda_device()
    if kind == "narrow":
        wl = wlmod.generate(wlmod.scaled(2, 300), 8080)
    else:
        wl = wlmod.generate(dict(num_ctx=5, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=700, rows_fixed=1600,
                                 dup_frac=0.0, density=0.5, n_contra=2), 8081)
    store = binding.Store(wl.n_bits, device=dev)
    state, status = _caller_state(store, dev)
    for ro, xo, xs, ys in _two_batches(wl):
        ro_t, xo_t, x_t, y_t = dev_arrays(binding, dev, ro, xo, xs, ys)
        store.learn(ro_t, x_t, xo_t, y_t)
        assert _noalloc_call(binding, wl.n_bits, state, status, ro_t, x_t, xo_t, y_t) == binding.F2_OK
        torch.cuda.synchronize()
        assert int(status.item()) == binding.F2_OK
        _compare(binding, store, state)
    assert store.device_status() == binding.F2_OK


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
