"""Learning and encoding from host memory (f2_learn_host, f2_encode_host):
chunked copies overlapped with the kernels give the oracle's results, with
chunks of a few contexts or queries, pinned or pageable host arrays,
incremental batches and feature rows stored out of context order."""
import numpy as np
import pytest
import torch

from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, cuda_device, lib, oracle_for

pytestmark = pytest.mark.gpu


def _pinned(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a).pin_memory()


def _assert_equal_to_oracle(binding, st, O):
    got = st.basis()
    torch.cuda.synchronize()
    ref = O.export()
    for k in KEYS:
        assert np.array_equal(as_bytes(binding.to_numpy(got[k])), as_bytes(ref[k])), k


@pytest.mark.parametrize("chunk", [1 << 16, 1 << 20, 128 << 20])
@pytest.mark.parametrize("pinned", [True, False])
def test_learn_host_matches_oracle(chunk, pinned):
    dev = cuda_device()
    binding = lib()
    wl = wlmod.generate(wlmod.scaled(2, 300), 4242)
    st = binding.Store(wl.n_bits, device=dev)
    st.set_option(binding.F2_OPT_HOST_CHUNK_BYTES, chunk)
    conv = _pinned if pinned else np.ascontiguousarray
    hx, hy = conv(wl.x), conv(wl.y)
    for ro, xo in wl.batches:
        st.learn_host(conv(ro), hx, conv(xo), hy)
    _assert_equal_to_oracle(binding, st, oracle_for(wl))
    st.close()


def test_learn_host_incremental_and_permuted_rows():
    """Two batches; the second stores the contexts' feature rows in reverse
    context order (x_off decreasing), so chunks gather non-monotone ranges."""
    dev = cuda_device()
    binding = lib()
    cfg = dict(num_ctx=40, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=100, rows_fixed=600, dup_frac=0.0,
               density=0.3, n_contra=4, batch_rows=300)
    wl = wlmod.generate(cfg, 77)
    assert len(wl.batches) == 2
    st = binding.Store(wl.n_bits, device=dev)
    st.set_option(binding.F2_OPT_HOST_CHUNK_BYTES, 1 << 16)
    ro1, xo1 = wl.batches[0]
    st.learn_host(_pinned(ro1), _pinned(wl.x), _pinned(xo1), _pinned(wl.y))
    # batch 2 rebuilt with the contexts' x blocks in reverse order
    ro2, xo2 = wl.batches[1]
    C = wl.num_ctx
    W = (wl.n_bits.astype(np.int64) + 31) // 32
    blocks = [wl.x[int(xo2[c]):int(xo2[c]) + int(ro2[c + 1] - ro2[c]) * int(W[c])] for c in range(C)]
    x2 = np.concatenate(blocks[::-1])
    xo2r = np.zeros(C, np.int64)
    pos = 0
    for c in range(C - 1, -1, -1):
        xo2r[c] = pos
        pos += len(blocks[c])
    st.learn_host(_pinned(ro2), _pinned(x2), _pinned(xo2r), _pinned(wl.y))
    _assert_equal_to_oracle(binding, st, oracle_for(wl))
    st.close()


def test_learn_host_rejects_bad_offsets():
    dev = cuda_device()
    binding = lib()
    st = binding.Store(np.array([8, 8], np.int32), device=dev)
    x = np.zeros(8, np.uint32)
    y = np.zeros((4, 4), np.uint32)
    for ro, xo in ((np.array([0, 3, 2], np.int64), np.array([0, 0], np.int64)),   # decreasing
                   (np.array([0, 2, 5], np.int64), np.array([0, 2], np.int64)),   # past total_rows
                   (np.array([0, 2, 4], np.int64), np.array([0, 7], np.int64))):  # x past the array
        with pytest.raises(binding.F2Error) as e:
            st.learn_host(ro, x, xo, y)
        assert e.value.code == 1
    st.close()


@pytest.mark.parametrize("chunk", [1 << 16, 128 << 20])
def test_encode_host_matches_device_and_oracle(chunk):
    dev = cuda_device()
    binding = lib()
    wl = wlmod.generate(wlmod.scaled(3, 800), 515, query_count=120000)
    st = binding.Store(wl.n_bits, device=dev)
    st.set_option(binding.F2_OPT_HOST_CHUNK_BYTES, chunk)
    for ro, xo in wl.batches:
        st.learn_host(_pinned(ro), _pinned(wl.x), _pinned(xo), _pinned(wl.y))
    q = wl.queries
    Q = len(q.ctx_id)
    hy = torch.zeros((Q, 4), dtype=torch.int32).pin_memory()
    hs = torch.zeros(Q, dtype=torch.uint8).pin_memory()
    st.encode_host(_pinned(q.ctx_id), _pinned(q.x), hy, hs)
    torch.cuda.synchronize()
    dy, ds = st.encode(binding.to_device(q.ctx_id, dev), binding.to_device(q.x, dev))
    torch.cuda.synchronize()
    assert np.array_equal(hy.numpy(), binding.to_numpy(dy).view(np.int32))
    assert np.array_equal(hs.numpy(), binding.to_numpy(ds))
    O = oracle_for(wl)
    oy, ok = O.encode(q.ctx_id, q.x)
    assert np.array_equal(hy.numpy().view(np.uint32), oy)
    assert np.array_equal(hs.numpy(), ok)
    assert 0 < int(ok.sum()) < Q
    assert st.device_status() == 0
    st.close()
