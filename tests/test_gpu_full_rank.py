"""Contexts that reach full rank (rank = d): later calls check every row
against T with no insertion (Sec. 2.2 steps (2)-(3)).  Bit-exact against
the oracle, with contradictions at the first row of a call, several in one
call, and after an earlier call already recorded one."""
import numpy as np
import pytest

import oracle

from gpu_util import assert_basis_equal, cuda_device, dev_arrays, lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    dev = cuda_device()
    return lib(), dev


def _batches(rng, n_bits, rows_per_batch, n_batches, raw, plant):
    """Uniform x, y from a planted affine (or linear, raw) map per context;
    plant[(c, batch)] = list of in-batch rows whose word gets one flipped bit."""
    C = len(n_bits)
    maps = []
    for n in n_bits:
        A = rng.integers(0, 2 ** 32, size=(n, 4), dtype=np.uint64).astype(np.uint32)
        b = np.zeros(4, np.uint32) if raw else rng.integers(0, 2 ** 32, size=4, dtype=np.uint64).astype(np.uint32)
        maps.append((A, b))
    out = []
    for bt in range(n_batches):
        xs, ys, row_off, x_off = [], [], [0], []
        pos = 0
        for c, n in enumerate(n_bits):
            W = (n + 31) // 32
            R = rows_per_batch[c]
            x = rng.integers(0, 2 ** 32, size=(R, W), dtype=np.uint64).astype(np.uint32)
            if n % 32:
                x[:, -1] &= np.uint32((1 << (n % 32)) - 1)
            bits = np.unpackbits(x.view(np.uint8), axis=1, bitorder="little")[:, :n].astype(bool)
            A, b = maps[c]
            y = np.tile(b, (R, 1))
            for j in range(n):
                y[bits[:, j]] ^= A[j]
            for r in plant.get((c, bt), []):
                y[r, rng.integers(4)] ^= np.uint32(1 << int(rng.integers(32)))
            x_off.append(pos)
            pos += R * W
            xs.append(x.reshape(-1))
            ys.append(y)
            row_off.append(row_off[-1] + R)
        out.append((np.array(row_off, np.int64), np.array(x_off, np.int64), np.concatenate(xs), np.concatenate(ys)))
    return out


@pytest.mark.parametrize("raw", [False, True])
@pytest.mark.parametrize("dedup", [1, 0])
def test_full_rank_calls(env, raw, dedup):
    import torch

    binding, dev = env
    rng = np.random.default_rng(11 + int(raw) + 2 * dedup)
    n_bits = [1, 5, 31, 32, 64, 95, 100, 200, 287, 300]
    d = [n if raw else n + 1 for n in n_bits]
    # batch 0 reaches full rank (uniform rows, a few more than d); the next
    # batches are checks only, of several chunk sizes
    rows = [[dd + 40 for dd in d], [3000] * len(d), [5000 + 17 * c for c in range(len(d))], [1] * len(d)]
    plant = {(2, 1): [0], (4, 1): [5, 2999], (4, 2): [0, 1, 4096], (7, 2): [2048], (9, 3): [0], (0, 1): [7]}
    batches = []
    for bt, rb in enumerate(rows):
        batches += _batches(rng, n_bits, rb, 1, raw, {(c, 0): v for (c, b), v in plant.items() if b == bt})
    st = binding.Store(n_bits, raw=raw, device=dev)
    st.set_option(binding.F2_OPT_DEDUP, dedup)
    O = oracle.Oracle(n_bits, raw=raw, threads=4)
    for ro, xo, x, y in batches:
        rt, xot, xt, yt = dev_arrays(binding, dev, ro, xo, x, y)
        st.learn(rt, xt, xot, yt)
        torch.cuda.synchronize()
        O.learn(ro, xo, x, y)
        assert_basis_equal(binding, st.basis(), O.export())
    ex = O.export()
    assert (ex["rank"] == np.array(d)).all()
    assert ex["contra"].sum() >= 5
    W = binding.to_numpy(st.solve()).view(np.uint32)
    assert np.array_equal(W, O.solve())
    assert st.device_status() == 0
