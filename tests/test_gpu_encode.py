"""Encode paths (Sec. 2.3) vs the CPU oracle: queries grouped by context,
long runs encoded with per-run lookup tables of the basis, the others by the
per-query pivot walk, and small passes with no grouping at all.  Every run
length, width and residual size that switches between the paths is covered,
with each path forced on and off."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import csr_from_rows, cuda_device, dev_arrays, gpu_learn_workload, lib, oracle_for

pytestmark = pytest.mark.gpu

TABLE_MINS = (16, 32, 200, 1 << 30)  # 1 << 30: tables off
DIRECT = "direct"  # every query on its own (F2_OPT_ENCODE_DIRECT_MAX above the pass)


@pytest.fixture(scope="module")
def env():
    dev = cuda_device()
    return lib(), dev


def _encode_all(binding, st, ctx, qx, table_min):
    if table_min == DIRECT:
        st.set_option(binding.F2_OPT_ENCODE_DIRECT_MAX, 1 << 30)
    else:  # the grouped path, whatever the pass size
        st.set_option(binding.F2_OPT_ENCODE_DIRECT_MAX, 0)
        st.set_option(binding.F2_OPT_ENCODE_TABLE_MIN, table_min)
    ct, xt = dev_arrays(binding, st.device, ctx, qx)
    y, ok = st.encode(ct, xt)
    torch.cuda.synchronize()
    return binding.to_numpy(y).view(np.uint32), binding.to_numpy(ok)


def _compare(binding, st, O, ctx, qx, expect_status=0):
    ry, rok = O.encode(ctx, qx)
    for tm in TABLE_MINS + (DIRECT,):
        y, ok = _encode_all(binding, st, ctx, qx, tm)
        bad = np.flatnonzero((ok != rok) | (y != ry).any(axis=1))
        assert bad.size == 0, (tm, bad[:8].tolist(), ctx[bad[:8]].tolist())
        assert st.device_status() == expect_status
    return ry, rok


def _run_lengths(rng, C, lengths):
    """Context ids: for each context a run of the given length, shuffled."""
    ids = np.concatenate([np.full(L, c, np.int32) for c, L in zip(range(C), lengths)])
    rng.shuffle(ids)
    return ids


@pytest.mark.parametrize("seed", range(3))
def test_run_lengths_and_widths(env, seed):
    """Widths 1..300 (tables up to d = 288), runs of 1..5000 queries (runs
    longer than one 2,048-query block), ranks from 0 to full."""
    binding, dev = env
    rng = np.random.default_rng(seed)
    n_bits = [1, 4, 31, 32, 63, 64, 65, 100, 127, 128, 200, 255, 256, 286, 287, 288, 300, 48, 48, 48]
    rows = [0, 3, 40, 10, 500, 64, 30, 1, 400, 100, 150, 800, 0, 500, 300, 600, 700, 200, 200, 5]
    # per context: a planted affine map observed on a random input subspace
    systems = []
    for c, (n, R) in enumerate(zip(n_bits, rows)):
        W = (n + 31) // 32
        k = int(rng.integers(1, n + 1))  # dimension of the planted input subspace
        basis = rng.integers(0, 2 ** 32, size=(k, W), dtype=np.uint64).astype(np.uint32)
        if n % 32:
            basis[:, -1] &= np.uint32((1 << (n % 32)) - 1)
        A = rng.integers(0, 2 ** 32, size=(n, 4), dtype=np.uint64).astype(np.uint32)
        b = rng.integers(0, 2 ** 32, size=4, dtype=np.uint64).astype(np.uint32)
        sys_rows = []
        for _ in range(R):
            sel = rng.random(k) < 0.5
            x = np.bitwise_xor.reduce(basis[sel], axis=0) if sel.any() else np.zeros(W, np.uint32)
            bits = np.unpackbits(x.view(np.uint8), bitorder="little")[:n].astype(bool)
            y = b ^ np.bitwise_xor.reduce(A[bits], axis=0) if bits.any() else b.copy()
            sys_rows.append((x, y))
        systems.append(sys_rows)
    ro, xo, x, y = csr_from_rows(n_bits, systems)
    st = binding.Store(n_bits, device=dev)

    rot, xot, xt, yt = dev_arrays(binding, dev, ro, xo, x, y)
    st.learn(rot, xt, xot, yt)
    torch.cuda.synchronize()
    O = oracle.Oracle(n_bits, threads=4)
    O.learn(ro, xo, x, y)
    lengths = [int(v) for v in rng.choice([1, 5, 15, 16, 17, 31, 32, 33, 100, 199, 200, 201, 2047, 2048, 2049,
                                           5000], size=len(n_bits))]
    ctx = _run_lengths(rng, len(n_bits), lengths)

    W = ((np.array(n_bits) + 31) // 32).max()
    qx = np.zeros((len(ctx), W), np.uint32)
    for i, c in enumerate(ctx):
        n = n_bits[c]
        w = (n + 31) // 32
        srows = systems[c]
        if srows and rng.random() < 0.7:
            v = srows[rng.integers(len(srows))][0].copy()
            if rng.random() < 0.5:
                v = v ^ srows[rng.integers(len(srows))][0]
            qx[i, :w] = v
        else:
            qx[i, :w] = rng.integers(0, 2 ** 32, size=w, dtype=np.uint64).astype(np.uint32)
    if seed % 2:  # rows padded to 16 bytes: the kernels' vector loads
        qx = np.ascontiguousarray(np.pad(qx, ((0, 0), (0, (-qx.shape[1]) % 4))))
    ry, rok = _compare(binding, st, O, ctx, qx)
    assert 0 < rok.mean() < 1


def test_raw_features_tables(env):
    """Raw feature rows (no affine constant): tables over d = n coordinates."""
    binding, dev = env
    rng = np.random.default_rng(7)
    n_bits = [8, 40, 96, 160, 256]
    systems = []
    for n in n_bits:
        W = (n + 31) // 32
        rows = []
        for _ in range(int(rng.integers(n // 2, 2 * n))):
            xw = rng.integers(0, 2 ** 32, size=W, dtype=np.uint64).astype(np.uint32)
            if n % 32:
                xw[-1] &= np.uint32((1 << (n % 32)) - 1)
            xw[0] &= np.uint32(0xFFFF0FFF)  # a few coordinates never set: non-pivots
            rows.append((xw, rng.integers(0, 2 ** 32, size=4, dtype=np.uint64).astype(np.uint32)))
        systems.append(rows)
    ro, xo, x, y = csr_from_rows(n_bits, systems)
    st = binding.Store(n_bits, raw=True, device=dev)
    rot, xot, xt, yt = dev_arrays(binding, dev, ro, xo, x, y)
    st.learn(rot, xt, xot, yt)
    torch.cuda.synchronize()
    O = oracle.Oracle(n_bits, raw=True, threads=2)
    O.learn(ro, xo, x, y)
    ctx = _run_lengths(rng, len(n_bits), [300, 64, 3000, 40, 500])
    W = 8
    qx = np.zeros((len(ctx), W), np.uint32)
    for i, c in enumerate(ctx):
        n = n_bits[c]
        w = (n + 31) // 32
        if rng.random() < 0.6:
            qx[i, :w] = systems[c][rng.integers(len(systems[c]))][0]
        else:
            qx[i, :w] = rng.integers(0, 2 ** 32, size=w, dtype=np.uint64).astype(np.uint32)
    _compare(binding, st, O, ctx, qx)


def test_bad_ids_and_stride_in_long_runs(env):
    """Out-of-range ids (a long run of them) and contexts wider than the
    query stride: 0xFF flags, zero words, the status recorded once."""
    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(2, 40), 808)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    rng = np.random.default_rng(3)
    narrow = np.flatnonzero(wl.n_bits <= 64).astype(np.int32)
    ctx = np.concatenate([np.repeat(narrow[:4], 300), np.full(700, wl.num_ctx, np.int32),
                          np.full(50, -3, np.int32)])
    rng.shuffle(ctx)
    qx = rng.integers(0, 2 ** 32, size=(len(ctx), 2), dtype=np.uint64).astype(np.uint32)
    y, ok = _compare(binding, st, O, ctx, qx, expect_status=3)
    assert (ok[ctx >= wl.num_ctx] == 0xFF).all() and (ok[ctx < 0] == 0xFF).all()
    wide = np.flatnonzero(wl.n_bits > 64).astype(np.int32)
    ctx2 = np.repeat(wide[:2], 100)
    for tm in TABLE_MINS + (DIRECT,):
        yy, ok2 = _encode_all(binding, st, ctx2, qx[:200], tm)
        assert (ok2 == 0xFF).all() and not yy.any()
        assert st.device_status() == 9


def test_zipf_config3_scaled_table_mins(env):
    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(3, 2000), 313, query_count=200000)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    _compare(binding, st, O, wl.queries.ctx_id, wl.queries.x)


def test_epilogue_appendix_c_on_gpu(env, golden_dir):
    """The Appendix C instruction end to end on the GPU: learn the five stored
    pairs of Table 6, encode the parsed values, merge scheduler control."""
    import json
    import os

    from oracle import f2_bigint as bi

    binding, dev = env
    with open(os.path.join(golden_dir, "appendix_c_hmma.json")) as f:
        g = json.load(f)
    d = g["feature_width"]

    def idx(t):
        return 0 if t == "const" else 1 + 64 * t[0] + t[1]

    rows = [(sum(1 << idx(t) for t in r["features"]), int(r["z"], 16)) for r in g["basis_rows"]]
    nw = (d + 31) // 32
    x = np.array([bi.int_to_words(r, nw) for r, _ in rows], np.uint32).reshape(-1)
    y = np.array([bi.int_to_words(z, 4) for _, z in rows], np.uint32)
    st = binding.Store([d], raw=True, device=dev)
    rt, xot, xt, yt = dev_arrays(binding, dev, np.array([0, 5], np.int64), np.array([0], np.int64), x, y)
    st.learn(rt, xt, xot, yt)
    f = bi.parsed_value_features(g["values"])
    ct, qt = dev_arrays(binding, dev, np.zeros(1, np.int32), np.array([bi.int_to_words(f, nw)], np.uint32))
    yq, ok = st.encode(ct, qt)
    sc = binding.to_device(np.array([int(g["sched_control"], 16)], np.int32), dev)
    st.encode_epilogue(ct, ok, yq, sched=sc)
    torch.cuda.synchronize()
    words = binding.to_numpy(yq).view(np.uint32)[0]
    assert bi.words_to_int(words) == int(g["y_full"], 16)
    assert words.astype("<u4").tobytes().hex(" ") == g["le_bytes"]


def test_epilogue_random(env):
    """Random control bits, recorded states and per-context opaque masks (the
    Appendix D mask, random masks, none) against the oracle's epilogue."""
    from oracle import f2_bigint as bi

    binding, dev = env
    wl = wlmod.generate(wlmod.scaled(3, 300), 77, query_count=30000)
    st = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, st, wl, dev)
    O = oracle_for(wl)
    q = wl.queries
    rng = np.random.default_rng(5)
    Q = len(q.ctx_id)
    ctx = q.ctx_id.copy()
    ctx[::997] = wl.num_ctx + 3  # a few bad ids: rejected, untouched
    sched = rng.integers(0, 2 ** 31, size=Q, dtype=np.int64).astype(np.int32)
    state = rng.integers(0, 2 ** 32, size=(Q, 4), dtype=np.uint64).astype(np.uint32)
    masks = np.zeros((wl.num_ctx, 4), np.uint32)
    masks[::3, 3] = (1 << (122 - 96)) | (1 << (124 - 96))
    masks[1::3] = rng.integers(0, 2 ** 32, size=masks[1::3].shape, dtype=np.uint64).astype(np.uint32)
    ry, rok = O.encode(ctx, q.x)
    ct, xt = dev_arrays(binding, dev, ctx, q.x)
    yq, ok = st.encode(ct, xt)
    for variant in ("all", "no_state", "no_sched"):
        y2 = yq.clone()
        st.encode_epilogue(ct, ok, y2, sched=None if variant == "no_sched" else binding.to_device(sched, dev),
                           state=None if variant == "no_state" else binding.to_device(state, dev),
                           opaque_mask=binding.to_device(masks, dev))
        torch.cuda.synchronize()
        got = binding.to_numpy(y2).view(np.uint32)
        assert np.array_equal(binding.to_numpy(ok), rok)
        for i in range(0, Q, 7):
            c = int(ctx[i])
            m = bi.words_to_int(masks[c]) if (0 <= c < wl.num_ctx and variant != "no_state") else 0
            want = bi.encode_epilogue(bi.words_to_int(ry[i]), rok[i] == 1,
                                      sched=0 if variant == "no_sched" else int(sched[i]) & 0xFFFFFFFF,
                                      state=bi.words_to_int(state[i]), mask=m)
            assert bi.words_to_int(got[i]) == want, (variant, i)
    st.device_status()
