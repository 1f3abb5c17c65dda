"""The learn, solve and encode calls captured in CUDA graphs and replayed
give the bits of eager calls (every call is stream-ordered: no host
synchronization, no allocation once the store's scratch has grown), on the
oracle-pinned small configuration with both width classes and a second
stream forked inside the learn call."""
import numpy as np
import pytest
import torch

from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, cuda_device, dev_arrays, lib

pytestmark = pytest.mark.gpu


def test_graph_replay_equals_eager():
    binding = lib()
    dev = cuda_device()
    wl = wlmod.generate(wlmod.scaled(3, 600), 3131, query_count=60_000)
    x_t, y_t = dev_arrays(binding, dev, wl.x, wl.y)
    bt = [dev_arrays(binding, dev, ro, xo) for ro, xo in wl.batches]
    ct, qt = dev_arrays(binding, dev, wl.queries.ctx_id, wl.queries.x)

    def run(st, W, y, ok):
        st.reset()
        for ro, xo in bt:
            st.learn(ro, x_t, xo, y_t)
        st.solve(out=W)
        st.encode(ct, qt, y, ok)

    outs = []
    for graph in (False, True):
        st = binding.Store(wl.n_bits, device=dev)
        W = torch.empty((int(st.slot_off[-1]), 4), dtype=torch.int32, device=dev)
        y = torch.empty((len(wl.queries.ctx_id), 4), dtype=torch.int32, device=dev)
        ok = torch.empty(len(wl.queries.ctx_id), dtype=torch.uint8, device=dev)
        run(st, W, y, ok)  # grows the scratch
        torch.cuda.synchronize()
        if graph:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, capture_error_mode="thread_local"):
                run(st, W, y, ok)
            W.zero_()
            y.zero_()
            ok.zero_()
            for _ in range(3):
                g.replay()
        else:
            run(st, W, y, ok)
        torch.cuda.synchronize()
        assert st.device_status() == binding.F2_OK
        b = st.basis()
        torch.cuda.synchronize()
        outs.append({**{k: as_bytes(binding.to_numpy(b[k])) for k in KEYS},
                     "W": binding.to_numpy(W).copy(), "y": binding.to_numpy(y).copy(), "ok": binding.to_numpy(ok).copy()})
        st.close()
    for k in outs[0]:
        assert np.array_equal(outs[0][k], outs[1][k]), k
