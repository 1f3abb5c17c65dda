"""Parsed-value contexts (Sec. 2.1: phi = [1 || bits64(v_0) || ...]) with the
paper's low exact-context ranks: the int64 values are passed to the library
as they are (zero-copy), and every output matches the oracle bit for bit."""
import numpy as np
import pytest
import torch

from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import assert_basis_equal, cuda_device, lib, oracle_for

pytestmark = pytest.mark.gpu


def test_parsed_lowrank_parity():
    dev = cuda_device()
    binding = lib()
    wl = wlmod.parsed_lowrank(num_ctx=600, seed=11)
    # the rows' k int64 values, as the caller holds them, viewed as uint32 words
    v64 = torch.from_numpy(wl.x.view(np.int64)).to(dev)
    x_t = v64.view(torch.int32)
    y_t = binding.to_device(wl.y, dev)
    ro, xo = (binding.to_device(a, dev) for a in wl.batches[0])
    st = binding.Store(wl.n_bits, device=dev)
    st.learn(ro, x_t, xo, y_t)
    torch.cuda.synchronize()
    O = oracle_for(wl)
    ex = O.export()
    assert_basis_equal(binding, st.basis(), ex)
    assert np.array_equal(binding.to_numpy(st.solve()).view(np.uint32), O.solve())
    assert np.median(ex["rank"]) <= 5 and np.array_equal(np.flatnonzero(ex["contra"]),
                                                         np.flatnonzero(wl.contra_pos >= 0))
    assert st.device_status() == 0
