"""Simulated device-allocation failures (the F2_OPT_FAIL_ALLOC test hook).

Every device allocation a call makes on a store goes through one helper, and
the hook makes the k-th one fail as if the device were out of memory.  For
every allocation site of each entry point (k = 0, 1, ... until the call
needs fewer allocations), the call must return F2_ERR_OOM and leave the store
usable: the same call again succeeds and gives the results of a store that
never failed.  Nothing here faults the GPU: the failure is made on the host.
"""
import numpy as np
import pytest
import torch

from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, cuda_device, dev_arrays, gpu_learn_workload, lib

pytestmark = pytest.mark.gpu

MAX_SITES = 40


@pytest.fixture(scope="module")
def env():
    dev = cuda_device()
    binding = lib()
    wl = wlmod.generate(wlmod.scaled(3, 200), 5151, query_count=20_000)
    ref = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, ref, wl, dev)
    q = wl.queries
    ct, qt = dev_arrays(binding, dev, q.ctx_id, q.x)
    y, ok = ref.encode(ct, qt)
    torch.cuda.synchronize()
    expect = {
        "basis": {k: as_bytes(binding.to_numpy(v)) for k, v in ref.basis().items()},
        "y": binding.to_numpy(y).copy(),
        "ok": binding.to_numpy(ok).copy(),
    }
    return binding, dev, wl, expect


def _same_basis(binding, st, expect):
    got = st.basis()
    torch.cuda.synchronize()
    for k in KEYS:
        assert np.array_equal(as_bytes(binding.to_numpy(got[k])), expect["basis"][k]), k


def _every_site(binding, make, call, check):
    """Fail the k-th allocation for k = 0, 1, ...: OOM, then the same call
    succeeds on the same store; returns how many sites failed."""
    for k in range(MAX_SITES):
        st = make()
        st.set_option(binding.F2_OPT_FAIL_ALLOC, k)
        try:
            call(st)
        except binding.F2Error as e:
            assert e.code == binding.F2_ERR_OOM, (k, e)
            torch.cuda.synchronize()
            call(st)  # the hook fired once and is off again
            check(st)
            st.close()
            continue
        # the call made fewer than k + 1 allocations: disarm before checking
        st.set_option(binding.F2_OPT_FAIL_ALLOC, -1)
        check(st)
        st.close()
        return k
    raise AssertionError("more allocation sites than expected")


def test_oom_learn(env):
    binding, dev, wl, expect = env
    x_t, y_t = dev_arrays(binding, dev, wl.x, wl.y)
    ro, xo = wl.batches[0]
    ro_t, xo_t = dev_arrays(binding, dev, ro, xo)

    def call(st):
        st.reset()
        st.learn(ro_t, x_t, xo_t, y_t)

    n = _every_site(binding, lambda: binding.Store(wl.n_bits, device=dev), call,
                    lambda st: _same_basis(binding, st, expect))
    assert n >= 2  # the duplicate pass's two per-row arrays


def test_oom_encode(env):
    binding, dev, wl, expect = env
    q = wl.queries
    ct, qt = dev_arrays(binding, dev, q.ctx_id, q.x)

    def make():
        st = binding.Store(wl.n_bits, device=dev)
        st.set_option(binding.F2_OPT_ENCODE_DIRECT_MAX, 0)  # the grouped path and its scratch
        gpu_learn_workload(binding, st, wl, dev)
        return st

    def check(st):
        y, ok = st.encode(ct, qt)
        torch.cuda.synchronize()
        assert np.array_equal(binding.to_numpy(y), expect["y"])
        assert np.array_equal(binding.to_numpy(ok), expect["ok"])

    n = _every_site(binding, make, lambda st: st.encode(ct, qt), check)
    assert n >= 7  # per-query scratch (3), buckets, per-context flags and offsets (2), table pool


def test_oom_host_paths(env):
    binding, dev, wl, expect = env
    ro, xo = wl.batches[0]
    q = wl.queries

    def learn(st):
        st.reset()
        st.learn_host(ro, wl.x, xo, wl.y)
        torch.cuda.synchronize()

    n = _every_site(binding, lambda: binding.Store(wl.n_bits, device=dev), learn,
                    lambda st: _same_basis(binding, st, expect))
    assert n >= 6  # two copy buffers of each kind, the CSR arrays, and the learn call's own

    def make():
        st = binding.Store(wl.n_bits, device=dev)
        gpu_learn_workload(binding, st, wl, dev)
        return st

    y = np.zeros((len(q.ctx_id), 4), np.uint32)
    ok = np.zeros(len(q.ctx_id), np.uint8)

    def encode(st):
        st.encode_host(q.ctx_id, q.x, y, ok)
        torch.cuda.synchronize()

    def check(st):
        encode(st)
        assert np.array_equal(y, expect["y"].view(np.uint32).reshape(y.shape))
        assert np.array_equal(ok, expect["ok"])

    n = _every_site(binding, make, encode, check)
    assert n >= 8


def test_oom_merge(env):
    binding, dev, wl, expect = env
    # groups of the most common width (members of a group share their width)
    widths, counts = np.unique(wl.n_bits, return_counts=True)
    same = np.flatnonzero(wl.n_bits == widths[np.argmax(counts)])
    G = min(8, len(same))
    group_of = np.full(wl.num_ctx, -1, np.int32)
    group_of[same] = np.arange(len(same)) % G
    base = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, base, wl, dev)
    merged_ref, ok_ref = base.merge(group_of, G)
    ref = {k: as_bytes(binding.to_numpy(v)) for k, v in merged_ref.basis().items()}
    torch.cuda.synchronize()

    def make():
        st = binding.Store(wl.n_bits, device=dev)
        gpu_learn_workload(binding, st, wl, dev)
        return st

    def check(st):
        merged, ok = st.merge(group_of, G)
        got = merged.basis()
        torch.cuda.synchronize()
        for k in KEYS:
            assert np.array_equal(as_bytes(binding.to_numpy(got[k])), ref[k]), k
        assert np.array_equal(ok, ok_ref)
        merged.close()

    n = _every_site(binding, make, lambda st: st.merge(group_of, G), check)
    assert n >= 6
