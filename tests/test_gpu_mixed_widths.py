"""One store holding contexts of every width class (feature rows of 1..3,
4..9, 10..17 and 18..33 words; dedup rows of up to 9 and of 10..16 words):
the kernels of disjoint classes run side by side on two streams, and the
result must still be the oracle's, bit for bit, through the device and the
host-memory entry points and over incremental calls."""
import numpy as np
import pytest
import torch

import oracle

from gpu_util import KEYS, as_bytes, csr_from_rows, cuda_device, lib

pytestmark = pytest.mark.gpu

WIDTHS = (5, 31, 64, 95, 96, 130, 200, 287, 288, 300, 350, 400, 511, 512, 544, 600, 800, 1000, 1024)


def _mixed(seed, n_ctx=57, batches=2):
    rng = np.random.default_rng(seed)
    n_bits = np.array([WIDTHS[c % len(WIDTHS)] for c in range(n_ctx)], np.int32)
    rows = [[[] for _ in range(n_ctx)] for _ in range(batches)]
    for c in range(n_ctx):
        n = int(n_bits[c])
        W = (n + 31) // 32
        r = int(rng.integers(1, min(n, 40) + 1))
        gens = rng.random((r, n)) < 0.4
        A = rng.random((n, 128)) < 0.1
        b = rng.random(128) < 0.5
        seen = []
        for bi in range(batches):
            for _ in range(int(rng.integers(0, 3 * r + 20))):
                if seen and rng.random() < 0.5:
                    xw, yw = seen[int(rng.integers(len(seen)))]  # a duplicate
                    yw = yw.copy()
                    if rng.random() < 0.01:
                        yw[int(rng.integers(4))] ^= np.uint32(1 << int(rng.integers(32)))  # contradiction
                else:
                    coef = rng.random(r) < 0.5
                    x = (coef.astype(np.int64) @ gens.astype(np.int64)) % 2 == 1
                    y = ((x.astype(np.int64) @ A.astype(np.int64)) % 2 == 1) ^ b
                    xw = np.pad(np.packbits(x, bitorder="little"), (0, 4 * W - (n + 7) // 8)).view(np.uint32)
                    yw = np.packbits(y, bitorder="little").view(np.uint32)
                    seen.append((xw, yw))
                rows[bi][c].append((xw, yw))
    return n_bits, [csr_from_rows(n_bits, rb) for rb in rows]


@pytest.mark.parametrize("host,all_cta", [(False, False), (True, False), (False, True)])
def test_every_width_class_in_one_store(host, all_cta):
    dev = cuda_device()
    binding = lib()
    n_bits, batches = _mixed(11)
    st = binding.Store(n_bits, device=dev)
    # all_cta: every context eliminated by a whole CTA (a store of 57 contexts
    # is that by default); else warps own every context whose basis fits
    st.set_option(binding.F2_OPT_HEAVY_ROWS, 1 if all_cta else 1 << 40)
    if host:
        st.set_option(binding.F2_OPT_HOST_CHUNK_BYTES, 1 << 16)
    O = oracle.Oracle(n_bits, threads=4)
    for ro, xo, x, y in batches:
        if host:
            st.learn_host(ro, x, xo, y)
        else:
            st.learn(*(binding.to_device(a, dev) for a in (ro, x, xo, y)))
        O.learn(ro, xo, x, y)
    got = st.basis()
    torch.cuda.synchronize()
    ref = O.export()
    for k in KEYS:
        assert np.array_equal(as_bytes(binding.to_numpy(got[k])), as_bytes(ref[k])), k
    assert ref["contra"].sum() > 0 and (ref["rank"] > 0).all()
    st.close()
