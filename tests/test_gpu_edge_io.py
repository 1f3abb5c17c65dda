"""Edge cases of the host-memory and pooling entry points: an empty batch,
one query, a query count just past the chunk minimum, pooling a raw-feature
store, and pooling into no groups."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, csr_from_rows, cuda_device, lib, oracle_for

pytestmark = pytest.mark.gpu


def _pinned(a):
    a = np.ascontiguousarray(a)
    return torch.from_numpy(a.view(np.int32) if a.dtype == np.uint32 else a).pin_memory()


def test_learn_host_empty_batch_changes_nothing():
    dev = cuda_device()
    binding = lib()
    wl = wlmod.generate(wlmod.scaled(2, 50), 61)
    st = binding.Store(wl.n_bits, device=dev)
    for ro, xo in wl.batches:
        st.learn_host(_pinned(ro), _pinned(wl.x), _pinned(xo), _pinned(wl.y))
    before = {k: binding.to_numpy(v).copy() for k, v in st.basis().items()}
    C = wl.num_ctx
    st.learn_host(np.zeros(C + 1, np.int64), np.zeros(1, np.uint32), np.zeros(C, np.int64),
                  np.zeros((1, 4), np.uint32))
    after = st.basis()
    torch.cuda.synchronize()
    for k in KEYS:
        assert np.array_equal(as_bytes(before[k]), as_bytes(binding.to_numpy(after[k]))), k
    st.close()


@pytest.mark.parametrize("Q", [1, 65537])
def test_encode_host_small_and_just_past_a_chunk(Q):
    dev = cuda_device()
    binding = lib()
    wl = wlmod.generate(wlmod.scaled(3, 300), 62, query_count=Q)
    st = binding.Store(wl.n_bits, device=dev)
    for ro, xo in wl.batches:
        st.learn(*(binding.to_device(a, dev) for a in (ro, wl.x, xo, wl.y)))
    q = wl.queries
    hy = torch.zeros((Q, 4), dtype=torch.int32).pin_memory()
    hs = torch.zeros(Q, dtype=torch.uint8).pin_memory()
    st.encode_host(_pinned(q.ctx_id), _pinned(q.x), hy, hs)
    torch.cuda.synchronize()
    O = oracle_for(wl)
    oy, ok = O.encode(q.ctx_id, q.x)
    assert np.array_equal(hy.numpy().view(np.uint32), oy)
    assert np.array_equal(hs.numpy(), ok)
    st.close()


@pytest.mark.parametrize("with_mask", [False, True])
def test_merge_raw_store(with_mask):
    dev = cuda_device()
    binding = lib()
    rng = np.random.default_rng(63)
    n_bits = np.array([40] * 6 + [70] * 6, np.int32)
    rows = []
    for c in range(len(n_bits)):
        n = int(n_bits[c])
        W = (n + 31) // 32
        A = rng.random((n, 128)) < 0.2
        k = []
        for _ in range(int(rng.integers(0, 12))):
            x = rng.random(n) < 0.3
            y = (x.astype(np.int64) @ A.astype(np.int64)) % 2 == 1
            xw = np.pad(np.packbits(x, bitorder="little"), (0, 4 * W - (n + 7) // 8)).view(np.uint32)
            k.append((xw, np.packbits(y, bitorder="little").view(np.uint32)))
        rows.append(k)
    ro, xo, x, y = csr_from_rows(n_bits, rows)
    st = binding.Store(n_bits, raw=True, device=dev)
    st.learn(*(binding.to_device(a, dev) for a in (ro, x, xo, y)))
    group_of = np.array([0, 0, 0, 1, 1, 1, 2, 2, 2, 3, 3, -1], np.int32)
    masks = None
    if with_mask:
        masks = np.full((len(n_bits), 4), 0xFFFFFFFF, np.uint32)
        masks[4, 3] = 0x0FFFFFFF
    merged, ok = st.merge(group_of, 4, out_mask=masks)
    got = merged.basis()
    torch.cuda.synchronize()
    O = oracle.Oracle(n_bits, raw=True, threads=2)
    O.learn(ro, xo, x, y)
    ex = O.export()
    dg = np.array([40, 40, 70, 70], np.int64)
    grp = [[] for _ in range(4)]
    for c in range(len(n_bits)):
        g = group_of[c]
        if g < 0:
            continue
        v = oracle.ctx_view(ex, O.layout, c)
        wd = (int(n_bits[c]) + 31) // 32
        for kk in range(int(n_bits[c])):
            if (int(v["pivot_mask"][kk // 32]) >> (kk % 32)) & 1:
                grp[g].append((np.array(v["basis_x"][kk][:wd], np.uint32), np.array(v["basis_z"][kk], np.uint32)))
    mro, mxo, mx, my = csr_from_rows(dg, grp)
    OM = oracle.Oracle(dg, raw=True, threads=2)
    OM.learn(mro, mxo, mx, my)
    ref = OM.export()
    for k in KEYS:
        assert np.array_equal(as_bytes(binding.to_numpy(got[k])), as_bytes(ref[k])), k
    assert ok.tolist() == ([1, 0, 1, 1] if with_mask else [1, 1, 1, 1])
    merged.close()
    st.close()


def test_merge_into_no_groups():
    dev = cuda_device()
    binding = lib()
    st = binding.Store(np.array([8, 8], np.int32), device=dev)
    merged, ok = st.merge(np.array([-1, -1], np.int32), 0)
    assert merged.num_ctx == 0 and len(ok) == 0
    merged.close()
    st.close()
