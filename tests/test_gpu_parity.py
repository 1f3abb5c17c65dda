"""CUDA path vs CPU oracle: bit-exact parity on paper examples, tiny random
systems, scaled workloads and edge cases, all through the C ABI."""
import json
import os
import random

import numpy as np
import pytest

import oracle
from oracle import f2_bigint as bi
from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import (KEYS, assert_basis_equal, csr_from_rows, cuda_device, dev_arrays, gpu_learn_workload, lib,
                      oracle_for)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    dev = cuda_device()
    return lib(), dev


def _learn_csr(binding, dev, n_bits, row_off, x_off, x, y, raw=False, options=None):
    import torch

    st = binding.Store(n_bits, raw=raw, device=dev)
    for k, v in (options or {}).items():
        st.set_option(k, v)
    ro, xo, xt, yt = dev_arrays(binding, dev, row_off, x_off, x, y)
    st.learn(ro, xt, xo, yt)
    torch.cuda.synchronize()
    return st


def _check_store(binding, st, O, queries=None):
    assert_basis_equal(binding, st.basis(), O.export())
    W = binding.to_numpy(st.solve()).view(np.uint32)
    assert np.array_equal(W, O.solve())
    if queries is not None:
        ctx, qx = queries
        import torch

        ct, xt = dev_arrays(binding, st.device, ctx, qx)
        y, ok = st.encode(ct, xt)
        ry, rok = O.encode(ctx, qx)
        assert np.array_equal(binding.to_numpy(ok), rok)
        assert np.array_equal(binding.to_numpy(y).view(np.uint32), ry)
    assert st.device_status() == 0


def test_appendix_b_on_gpu(env, golden_dir):
    binding, dev = env
    with open(os.path.join(golden_dir, "appendix_b_trace.json")) as f:
        g = json.load(f)
    rows = [(np.array([int(q, 2)], np.uint32), np.array([int(y, 2), 0, 0, 0], np.uint32))
            for q, y in g["observations"]]
    ro, xo, x, y = csr_from_rows([4], [rows])
    st = _learn_csr(binding, dev, [4], ro, xo, x, y, raw=True)
    b = st.basis()
    bx = binding.to_numpy(b["basis_x"]).view(np.uint32)
    bz = binding.to_numpy(b["basis_z"]).view(np.uint32)
    want = {int(k): (int(r, 2), int(z, 2)) for k, (r, z) in g["final_basis"].items()}
    got = {k: (int(bx[k]), int(bz[k][0])) for k in range(4) if bx[k]}
    assert got == want
    assert int(binding.to_numpy(b["rank"])[0]) == 3
    qx = np.array([[int(g["encode_supported"]["query"], 2)], [int(g["encode_rejected"]["query"], 2)]], np.uint32)
    ct, xt = dev_arrays(binding, dev, np.zeros(2, np.int32), qx)
    yq, ok = st.encode(ct, xt)
    assert binding.to_numpy(ok).tolist() == [1, 0]
    yq = binding.to_numpy(yq).view(np.uint32)
    assert int(yq[0][0]) == int(g["encode_supported"]["word"], 2) and not yq[1].any()


def test_appendix_c_wide_raw_on_gpu(env, golden_dir):
    """d = 321 raw features: exercises the wide (d > 288) kernels."""
    binding, dev = env
    with open(os.path.join(golden_dir, "appendix_c_hmma.json")) as f:
        g = json.load(f)
    d = g["feature_width"]
    idx = lambda t: 0 if t == "const" else 1 + 64 * t[0] + t[1]
    nw = (d + 31) // 32
    rows = [(np.array(bi.int_to_words(sum(1 << idx(t) for t in r["features"]), nw), np.uint32),
             np.array(bi.int_to_words(int(r["z"], 16), 4), np.uint32)) for r in g["basis_rows"]]
    ro, xo, x, y = csr_from_rows([d], [rows])
    st = _learn_csr(binding, dev, [d], ro, xo, x, y, raw=True)
    f = bi.parsed_value_features(g["values"])
    qx = np.array([bi.int_to_words(f, nw), bi.int_to_words(f ^ 1, nw)], np.uint32)
    ct, xt = dev_arrays(binding, dev, np.zeros(2, np.int32), qx)
    yq, ok = st.encode(ct, xt)
    assert binding.to_numpy(ok).tolist() == [1, 0]
    assert bi.words_to_int(binding.to_numpy(yq).view(np.uint32)[0]) == int(g["y_learned"], 16)
    O = oracle.Oracle([d], raw=True, threads=1)
    O.learn(ro, xo, x, y)
    _check_store(binding, st, O)


def _random_tiny(seed, C=64):
    rng = random.Random(seed)
    ds, systems = [], []
    for c in range(C):
        d = rng.randint(1, 12)
        M = [rng.getrandbits(128) for _ in range(d)]
        rows = []
        for i in range(rng.randint(0, 40)):
            if rows and rng.random() < 0.4:
                r = bi.words_to_int(rows[rng.randrange(len(rows))][0])
            else:
                r = rng.getrandbits(d)
            z = 0
            for j in range(d):
                if (r >> j) & 1:
                    z ^= M[j]
            if rng.random() < 0.05:
                z ^= 1 << rng.randrange(128)
            rows.append((np.array([r], np.uint32), np.array(bi.int_to_words(z, 4), np.uint32)))
        ds.append(d)
        systems.append(rows)
    return ds, systems


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("mode", ["warp", "cta"])
def test_tiny_random_systems(env, seed, mode):
    binding, dev = env
    ds, systems = _random_tiny(seed)
    ro, xo, x, y = csr_from_rows(ds, systems)
    # a store this small gives every context a CTA unless the threshold is set
    opts = {binding.F2_OPT_HEAVY_ROWS: 1 if mode == "cta" else 1 << 40}
    st = _learn_csr(binding, dev, ds, ro, xo, x, y, raw=True, options=opts)
    O = oracle.Oracle(ds, raw=True, threads=1)
    O.learn(ro, xo, x, y)
    qs = np.array([[random.Random(seed * 7 + i).getrandbits(12)] for i in range(4000)], np.uint32)
    ctx = np.array([i % len(ds) for i in range(4000)], np.int32)
    qs &= np.array([(1 << ds[c]) - 1 for c in ctx], np.uint32)[:, None]
    _check_store(binding, st, O, queries=(ctx, qs))


def test_config1(env):
    binding, dev = env
    wl = wlmod.standard(1)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    _check_store(binding, st, O, queries=(wl.queries.ctx_id, wl.queries.x))
    ex = O.export()
    assert np.array_equal(np.flatnonzero(ex["contra"]), np.flatnonzero(wl.contra_pos >= 0))


@pytest.mark.parametrize("mode", ["default", "all_cta", "all_warp", "cta4", "all_cta4"])
def test_config2_scaled(env, mode):
    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(2, 400), 202)
    st = binding.Store(wl.n_bits, device=dev)
    if mode in ("cta4", "all_cta4"):  # the 4..9-word contexts' CTAs of four warps
        st.set_option(binding.F2_OPT_LONG_CALL_ROWS, 0)
    if mode in ("all_cta", "all_cta4"):
        st.set_option(binding.F2_OPT_HEAVY_ROWS, 1)
    if mode == "all_warp":
        st.set_option(binding.F2_OPT_HEAVY_ROWS, 1 << 40)
        st.set_option(binding.F2_OPT_WARP_WORK, 1 << 50)
        st.set_option(binding.F2_OPT_WARP_BASIS_BYTES, 24576)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    q = wlmod.make_queries(wl, dict(ctx_mode=1, count=20000, zipf_s=1.1, out_frac=0.05), 99)
    _check_store(binding, st, O, queries=(q.ctx_id, q.x))


@pytest.mark.parametrize("shards", [1, 2, 3, 8])
def test_dedup_shards(env, shards):
    """Contexts far above their share of a call's rows have their duplicate
    pass split over several CTAs (F2_OPT_DEDUP_SHARDS at most): a row equal
    to one of an earlier shard is then classified by the elimination instead,
    and every exported array, the solve and the encode stay the oracle's."""
    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(2, 48, rows_median=3000, rows_max=40000, n_contra=6), 2024)
    assert int(wl.rows.max()) > 16384  # split 8 ways: far above 1/(4 x SMs) of the rows
    st = binding.Store(wl.n_bits, device=dev)
    st.set_option(binding.F2_OPT_DEDUP_SHARDS, shards)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    q = wlmod.make_queries(wl, dict(ctx_mode=1, count=20000, zipf_s=1.1, out_frac=0.05), 98)
    _check_store(binding, st, O, queries=(q.ctx_id, q.x))


def _affine_rows(rng, n, T, r1, late_new, contra_at):
    """T observations of one context: x in the span of r1 random generators
    (two more from row 0.8 T on when late_new), half of them repeats of
    earlier rows, y a planted affine map of x, and the rows in contra_at
    repeats of earlier rows with one flipped word bit (contradictions)."""
    W = (n + 31) // 32
    def rand_vec(k):
        v = rng.integers(0, 2 ** 32, size=(k, W), dtype=np.uint64).astype(np.uint32)
        if n % 32:
            v[:, -1] &= np.uint32((1 << (n % 32)) - 1)
        return v
    gens, late = rand_vec(r1), rand_vec(2)
    coef = rng.random((T, r1)) < 0.5
    x = np.zeros((T, W), np.uint32)
    for j in range(r1):
        x ^= gens[j] * coef[:, j:j + 1].astype(np.uint32)
    if late_new:
        lo = int(0.8 * T)
        for j in range(2):
            x[lo:] ^= late[j] * (rng.random((T - lo, 1)) < 0.5).astype(np.uint32)
    cols = rng.integers(0, 2 ** 32, size=(n + 1, 4), dtype=np.uint64).astype(np.uint32)
    def word(xr):
        yv = cols[0].copy()
        for j in range(n):
            if (int(xr[j // 32]) >> (j % 32)) & 1:
                yv ^= cols[1 + j]
        return yv
    y = np.stack([word(x[i]) for i in range(T)])
    for i in range(1, T):  # repeats of earlier rows
        if rng.random() < 0.5:
            k = int(rng.integers(0, i))
            x[i], y[i] = x[k], y[k]
    for i in contra_at:
        k = int(rng.integers(0, i))
        x[i], y[i] = x[k], y[k].copy()
        y[i][0] ^= np.uint32(1)
    return [(x[i], y[i]) for i in range(T)]


@pytest.mark.parametrize("late_new", [False, True])
def test_handoff_check_and_resume(env, late_new):
    """A CTA-owned context whose rank stops growing hands the rest of its
    rows off to the parallel check (F2_OPT_HANDOFF_REPS); with late_new a
    row outside the basis turns up there and sends the rest back to
    elimination from that row.  Contradictions before and after that point;
    every exported array and the solve equal the oracle's."""
    binding, dev = env
    rng = np.random.default_rng(4242 + int(late_new))
    n_bits = [20, 40, 70, 100, 150, 260, 400]
    T = 3000
    systems = [_affine_rows(rng, n, T, int(rng.integers(3, 12)), late_new, [900, 2700]) for n in n_bits]
    ro, xo, x, y = csr_from_rows(n_bits, systems)
    for opts in ({binding.F2_OPT_HEAVY_ROWS: 1, binding.F2_OPT_HANDOFF_REPS: 256},
                 {binding.F2_OPT_HEAVY_ROWS: 1, binding.F2_OPT_HANDOFF_REPS: 256, binding.F2_OPT_DEDUP: 0},
                 {binding.F2_OPT_HEAVY_ROWS: 1, binding.F2_OPT_HANDOFF_REPS: 0}):
        st = _learn_csr(binding, dev, n_bits, ro, xo, x, y, options=opts)
        O = oracle.Oracle(n_bits, threads=2)
        O.learn(ro, xo, x, y)
        _check_store(binding, st, O)
        ex = O.export()
        assert ex["contra"].all()  # both planted contradictions in every context
        st.close()


def test_config3_scaled(env):
    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(3, 1500), 303, query_count=50000)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    _check_store(binding, st, O, queries=(wl.queries.ctx_id, wl.queries.x))
    assert int(binding.to_numpy(st.basis()["contra"]).sum()) == 0


def test_config5_scaled_incremental(env):
    """n = 1024 (d = 1025, the widest row), batch-major incremental calls."""
    binding, dev = env
    cfg = dict(num_ctx=6, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=1024, rows_fixed=4096, dup_frac=0.0,
               density=0.5, n_contra=3, batch_rows=1024)
    wl = wlmod.generate(cfg, 505)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    _check_store(binding, st, O)
    ex = O.export()
    assert np.array_equal(ex["first_contra"][wl.contra_pos >= 0], wl.contra_pos[wl.contra_pos >= 0])


@pytest.mark.parametrize("n", [1, 31, 32, 33, 63, 64, 65, 127, 128, 255, 256, 287, 288, 300, 511, 1023, 1024])
def test_width_boundaries(env, n):
    binding, dev = env
    cfg = dict(num_ctx=5, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=n, rows_fixed=max(8, min(3 * n, 1500)),
               dup_frac=0.0, density=0.3, n_contra=2)
    wl = wlmod.generate(cfg, 1000 + n)
    for opts in ({}, {binding.F2_OPT_HEAVY_ROWS: 1 << 40}):  # (five contexts: a CTA each by default)
        st = binding.Store(wl.n_bits, device=dev)
        for k, v in opts.items():
            st.set_option(k, v)
        gpu_learn_workload(binding, st, wl, dev)
        O = oracle_for(wl)
        rng = np.random.default_rng(n)
        W = (n + 31) // 32
        qx = rng.integers(0, 2 ** 32, size=(300, W), dtype=np.uint64).astype(np.uint32)
        xs, _ = wl.ctx_rows(0)
        qx[:100] = xs[rng.integers(0, len(xs), 100)]
        _check_store(binding, st, O, queries=(np.zeros(300, np.int32) + (np.arange(300) % 5).astype(np.int32), qx))


def test_edge_cases(env):
    """Empty contexts, single rows, all-duplicate streams, a contradiction at
    the earliest possible row, rows of zeros."""
    binding, dev = env
    n_bits = [10, 10, 10, 10, 40, 3]
    one = np.array([0b1011001101], np.uint32)
    y1 = np.array([1, 2, 3, 4], np.uint32)
    rows = [
        [],                                    # empty context
        [(one, y1)],                           # one row
        [(one, y1)] * 50,                      # all duplicates
        [(one, y1), (one, y1 ^ np.array([0, 0, 0, 1 << 31], np.uint32))] + [(one, y1)] * 3,  # contradiction at row 1
        [(np.zeros(2, np.uint32), np.zeros(4, np.uint32))] * 5 + [(np.zeros(2, np.uint32), y1)],  # x = 0 rows
        [(np.array([7], np.uint32), y1), (np.array([15], np.uint32), y1 ^ np.array([1, 0, 0, 0], np.uint32))],  # bits above n ignored
    ]
    ro, xo, x, y = csr_from_rows(n_bits, rows)
    for opts in ({}, {binding.F2_OPT_HEAVY_ROWS: 1 << 40}):  # (six contexts: a CTA each by default)
        st = _learn_csr(binding, dev, n_bits, ro, xo, x, y, options=opts)
        O = oracle.Oracle(n_bits, threads=1)
        O.learn(ro, xo, x, y)
        _check_store(binding, st, O)
        ex = O.export()
        assert ex["first_contra"].tolist() == [-1, -1, -1, 1, 5, 1]
        assert ex["n_contra"].tolist() == [0, 0, 0, 1, 1, 1]


def test_incremental_equals_oracle_and_checkpoint(env):
    binding, dev = env
    import torch

    wl = wlmod.generate(wlmod.scaled(2, 120), 77)
    C = wl.num_ctx
    Wc = (wl.n_bits.astype(np.int64) + 31) // 32
    parts = []
    for part in range(3):
        lo = wl.row_off[:-1] + (wl.rows * part) // 3
        hi = wl.row_off[:-1] + (wl.rows * (part + 1)) // 3
        cnt = hi - lo
        ro = np.zeros(C + 1, np.int64)
        ro[1:] = np.cumsum(cnt)
        xs = np.concatenate([wl.x[wl.x_off[c] + (lo[c] - wl.row_off[c]) * Wc[c]:
                                  wl.x_off[c] + (hi[c] - wl.row_off[c]) * Wc[c]] for c in range(C)])
        xo = np.zeros(C, np.int64)
        xo[1:] = np.cumsum(cnt * Wc)[:-1]
        ys = np.concatenate([wl.y[lo[c]:hi[c]] for c in range(C)])
        parts.append((ro, xo, xs, ys))
    st = binding.Store(wl.n_bits, device=dev)
    O = oracle.Oracle(wl.n_bits, threads=2)
    for i, (ro, xo, xs, ys) in enumerate(parts):
        a, b, c_, d_ = dev_arrays(binding, dev, ro, xo, xs, ys)
        st.learn(a, c_, b, d_)
        O.learn(ro, xo, xs, ys)
        torch.cuda.synchronize()
        if i == 1:  # checkpoint after two batches, resume in a fresh store
            blob = st.export_state()
            st2 = binding.Store(wl.n_bits, device=dev)
            st2.import_state(blob)
            st.close()
            st = st2
    _check_store(binding, st, O)
    st.reset()
    assert int(binding.to_numpy(st.basis()["rank"]).sum()) == 0


def test_device_errors(env):
    binding, dev = env
    import torch

    n_bits = [8, 8]
    rows = [[(np.array([3], np.uint32), np.array([1, 0, 0, 0], np.uint32))]] * 2
    ro, xo, x, y = csr_from_rows(n_bits, rows)
    bad = ro.copy()
    bad[1] = 5  # context 0 claims rows past the end, context 1 goes backwards
    st = _learn_csr(binding, dev, n_bits, bad, xo, x, y)
    assert st.device_status() == binding.F2_ERR_ROWS
    assert binding.to_numpy(st.basis()["rows_seen"]).tolist() == [0, 0]
    ro_t, x_t, xo_t, y_t = dev_arrays(binding, dev, ro, x, xo, y)
    st.learn(ro_t, x_t, xo_t, y_t)
    assert st.device_status() == 0
    ct, qt = dev_arrays(binding, dev, np.array([0, 7, -1], np.int32), np.array([[3], [3], [3]], np.uint32))
    yq, ok = st.encode(ct, qt)
    torch.cuda.synchronize()
    assert binding.to_numpy(ok).tolist() == [1, 0xFF, 0xFF]
    assert st.device_status() == binding.F2_ERR_CTX_RANGE
    st2 = binding.Store([40], device=dev)
    ct, qt = dev_arrays(binding, dev, np.array([0], np.int32), np.array([[3]], np.uint32))
    _, ok = st2.encode(ct, qt)
    assert binding.to_numpy(ok).tolist() == [0xFF]
    assert st2.device_status() == binding.F2_ERR_STRIDE
    with pytest.raises(binding.F2Error):
        binding.Store([0], device=dev)


def test_deterministic(env):
    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(3, 300), 31)
    outs = []
    for _ in range(2):
        st = binding.Store(wl.n_bits, device=dev)
        gpu_learn_workload(binding, st, wl, dev)
        outs.append({k: binding.to_numpy(v).copy() for k, v in st.basis().items()})
    for k in KEYS:
        assert np.array_equal(outs[0][k], outs[1][k])
