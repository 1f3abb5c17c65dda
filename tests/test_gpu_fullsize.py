"""Parity at the benchmark sizes, in the launch configuration bench.py times.

Config 2 (4,096 contexts) and config 3 (77,926 contexts, ~81M rows) are
compared with the CPU oracle on every output; config 4's 10M queries are
encoded by both.  Config 5 (64 contexts, n = 1024, 2^20 rows each in 16
incremental calls) is compared on every context the oracle can replay in a
few seconds: all contradiction contexts and a sample of clean ones.
"""
import numpy as np
import pytest

import oracle
from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import (assert_basis_equal, assert_contexts_equal, cuda_device, gpu_learn_workload, lib, oracle_for,
                      oracle_for_contexts)

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def env():
    dev = cuda_device()
    return lib(), dev


def _encode_compare(binding, st, O, ctx, qx, chunk=2_000_000):
    import torch

    for a in range(0, len(ctx), chunk):
        c = ctx[a:a + chunk]
        x = qx[a:a + chunk]
        ct, xt = binding.to_device(c, st.device), binding.to_device(x, st.device)
        y, ok = st.encode(ct, xt)
        torch.cuda.synchronize()
        ry, rok = O.encode(c, x)
        assert np.array_equal(binding.to_numpy(ok), rok)
        assert np.array_equal(binding.to_numpy(y).view(np.uint32), ry)


def test_config2_full(env):
    binding, dev = env
    wl = wlmod.standard(2)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    ref = O.export()
    assert_basis_equal(binding, st.basis(), ref)
    assert np.array_equal(binding.to_numpy(st.solve()).view(np.uint32), O.solve())
    q = wlmod.make_queries(wl, dict(ctx_mode=1, count=200_000, zipf_s=1.1, out_frac=0.05), 2)
    _encode_compare(binding, st, O, q.ctx_id, q.x)
    injected = np.flatnonzero(wl.contra_pos >= 0)
    assert len(injected) == 20
    assert np.array_equal(np.flatnonzero(ref["contra"]), injected)
    assert st.device_status() == 0


def test_config3_and_4_full(env):
    binding, dev = env
    wl = wlmod.standard(3)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    ref = O.export()
    assert_basis_equal(binding, st.basis(), ref)
    assert int(ref["contra"].sum()) == 0
    assert np.array_equal(binding.to_numpy(st.solve()).view(np.uint32), O.solve())
    q = wl.queries
    assert len(q.ctx_id) == 10_000_000
    _encode_compare(binding, st, O, q.ctx_id, q.x)
    # the planted split: out-of-span constructions are rejected, in-span accepted
    ct, xt = binding.to_device(q.ctx_id[:1_000_000], dev), binding.to_device(q.x[:1_000_000], dev)
    _, ok = st.encode(ct, xt)
    assert np.array_equal(binding.to_numpy(ok), q.expect_in[:1_000_000])
    assert st.device_status() == 0


def test_config5_full_sampled(env):
    binding, dev = env
    wl = wlmod.standard(5)
    assert len(wl.batches) == 16
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    injected = np.flatnonzero(wl.contra_pos >= 0)
    clean = np.flatnonzero(wl.contra_pos < 0)[:4]
    sample = np.concatenate([injected, clean])
    O, ref = oracle_for_contexts(wl, sample)
    got = st.basis()
    assert_contexts_equal(binding, got, st, ref, O.layout, sample)
    # every context: full rank, rows seen, and exactly the injected contradiction
    rank = binding.to_numpy(got["rank"])
    assert np.all(rank == 1025)
    assert np.all(binding.to_numpy(got["rows_seen"]) == 1 << 20)
    first = binding.to_numpy(got["first_contra"])
    assert np.array_equal(first[injected], wl.contra_pos[injected])
    assert np.all(first[wl.contra_pos < 0] == -1)
    assert np.all(binding.to_numpy(got["n_contra"]) == (wl.contra_pos >= 0))
    # full rank: the solved map is the planted one, on every context (a
    # flipped word repeats an earlier row, so it is never inserted and the
    # contradicted contexts keep the planted map too)
    W = binding.to_numpy(st.solve()).view(np.uint32)
    for c in range(wl.num_ctx):
        s0 = int(st.slot_off[c])
        assert np.array_equal(W[s0], wl.b[c])
        assert np.array_equal(W[s0 + 1:s0 + 1025], wl.A[int(wl.a_off[c]):int(wl.a_off[c]) + 1024])
    assert st.device_status() == 0
