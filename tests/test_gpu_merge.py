"""Map pooling on the GPU (f2_merge_bases) against the oracle: groups of
exact contexts that share a planted map merge consistently; a group with a
foreign member is flagged; output masks are compared per group."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20532_gb300 import workloads as wlmod

from gpu_util import KEYS, as_bytes, cuda_device, gpu_learn_workload, lib, oracle_for

pytestmark = pytest.mark.gpu


def _export_rows(ex, layout, c, d):
    """Context c's basis rows (x words, z) in increasing pivot order."""
    v = oracle.ctx_view(ex, layout, c)
    wd = (d + 31) // 32
    out = []
    for k in range(d):
        if (int(v["pivot_mask"][k // 32]) >> (k % 32)) & 1:
            out.append((np.array(v["basis_x"][k][:wd], np.uint32), np.array(v["basis_z"][k], np.uint32)))
    return out


def test_merge_parity():
    dev = cuda_device()
    binding = lib()
    wl = wlmod.parsed_lowrank(num_ctx=240, seed=21, group_size=6, rows_per_rank=30)
    C = wl.num_ctx
    st = binding.Store(wl.n_bits, device=dev)
    x_t, y_t = binding.to_device(wl.x, dev), binding.to_device(wl.y, dev)
    ro, xo = (binding.to_device(a, dev) for a in wl.batches[0])
    st.learn(ro, x_t, xo, y_t)
    torch.cuda.synchronize()
    # groups of the workload, plus some contexts moved to a foreign group of
    # the same width, and some left out
    group_of = np.arange(C, dtype=np.int32) // 6
    G = int(group_of.max()) + 1
    rng = np.random.default_rng(4)
    for c in rng.choice(C, 12, replace=False):
        same = np.flatnonzero((wl.n_bits == wl.n_bits[c]) & (group_of // 1 != group_of[c]))
        if len(same):
            group_of[c] = group_of[rng.choice(same)]
    group_of[rng.choice(C, 5, replace=False)] = -1
    present = np.unique(group_of[group_of >= 0])
    remap = -np.ones(G, np.int32)
    remap[present] = np.arange(len(present), dtype=np.int32)
    group_of = np.where(group_of >= 0, remap[np.maximum(group_of, 0)], -1).astype(np.int32)
    G = len(present)
    masks = np.tile(np.array([0xFFFFFFFF, 0xFFFFFFFF, 0xFFFFFFFF, 0xEBFFFFFF], np.uint32), (C, 1))
    masks[rng.choice(C, 7, replace=False), 3] = 0xFFFFFFFF  # some contexts keep bits 122/124
    merged, mask_ok = st.merge(group_of, G, out_mask=masks)
    got = merged.basis()
    torch.cuda.synchronize()
    # oracle: learn the workload, then the members' rows of each group as one stream
    O = oracle_for(wl)
    ex = O.export()
    d = (wl.n_bits + 1).astype(np.int64)
    dg = np.zeros(G, np.int64)
    rows = [[] for _ in range(G)]
    for c in range(C):
        g = group_of[c]
        if g >= 0:
            dg[g] = d[c]
            rows[g] += _export_rows(ex, O.layout, c, int(d[c]))
    from gpu_util import csr_from_rows

    mro, mxo, mx, my = csr_from_rows(dg, rows)
    OM = oracle.Oracle(dg, raw=True, threads=4)
    OM.learn(mro, mxo, mx, my)
    ref = OM.export()
    g_np = {k: binding.to_numpy(got[k]) for k in KEYS}
    for k in KEYS:
        assert np.array_equal(as_bytes(g_np[k]), as_bytes(ref[k])), k
    assert ref["contra"].sum() > 0 and (ref["contra"] == 0).sum() > 0
    want_ok = np.ones(G, np.uint8)
    for g in range(G):
        mem = np.flatnonzero(group_of == g)
        if (masks[mem] != masks[mem[0]]).any():
            want_ok[g] = 0
    assert np.array_equal(mask_ok, want_ok) and (want_ok == 0).any()
    merged.close()


def _overlap_store(rng, raw, n_groups=40, gs=5):
    """Groups of gs contexts of one width whose input spans overlap (random
    combinations of a shared generator set); y is a shared map of x, except
    for one member of every third group, which sees a map that differs in one
    column.  Some members get no rows."""
    widths = [8, 31, 64, 100, 257, 600]
    n_bits, rows, foreign = [], [], []
    for g in range(n_groups):
        n = widths[g % len(widths)]
        r = int(rng.integers(1, min(n, 24) + 1))
        gens = rng.random((r, n)) < 0.3
        A = rng.random((n, 128)) < 0.2
        b = rng.random(128) < 0.5
        for m in range(gs):
            Am = A.copy()
            bad = g % 3 == 0 and m == gs - 1
            if bad:
                Am[int(rng.integers(n))] ^= True
            cnt = 0 if rng.random() < 0.1 else int(rng.integers(1, 2 * r + 2))
            coef = rng.random((cnt, r)) < 0.5
            X = (coef.astype(np.int64) @ gens.astype(np.int64)) % 2 == 1
            Y = ((X.astype(np.int64) @ Am.astype(np.int64)) % 2 == 1) ^ (False if raw else b)
            Xw = np.packbits(X, axis=1, bitorder="little") if cnt else np.zeros((0, (n + 7) // 8), np.uint8)
            W = (n + 31) // 32
            Xw = np.pad(Xw, ((0, 0), (0, 4 * W - Xw.shape[1]))).view(np.uint32)
            Yw = np.packbits(Y, axis=1, bitorder="little").view(np.uint32) if cnt else np.zeros((0, 4), np.uint32)
            rows.append([(Xw[i], Yw[i]) for i in range(cnt)])
            n_bits.append(n)
            foreign.append(bad)
    return np.array(n_bits, np.int32), rows, np.array(foreign)


@pytest.mark.parametrize("raw", [False, True])
def test_merge_parity_overlapping_spans(raw):
    dev = cuda_device()
    binding = lib()
    rng = np.random.default_rng(77 + raw)
    gs = 5
    n_bits, rows, foreign = _overlap_store(rng, raw, gs=gs)
    from gpu_util import csr_from_rows

    ro, xo, x, y = csr_from_rows(n_bits, rows)
    C = len(n_bits)
    st = binding.Store(n_bits, raw=raw, device=dev)
    st.learn(*(binding.to_device(a, dev) for a in (ro, x, xo, y)))
    group_of = (np.arange(C) // gs).astype(np.int32)
    G = C // gs
    merged, mask_ok = st.merge(group_of, G)
    got = merged.basis()
    torch.cuda.synchronize()
    O = oracle.Oracle(n_bits, raw=raw, threads=4)
    O.learn(ro, xo, x, y)
    ex = O.export()
    d = n_bits.astype(np.int64) + (0 if raw else 1)
    dg = d[::gs]
    grp = [[] for _ in range(G)]
    for c in range(C):
        grp[c // gs] += _export_rows(ex, O.layout, c, int(d[c]))
    mro, mxo, mx, my = csr_from_rows(dg, grp)
    OM = oracle.Oracle(dg, raw=True, threads=4)
    OM.learn(mro, mxo, mx, my)
    ref = OM.export()
    for k in KEYS:
        assert np.array_equal(as_bytes(binding.to_numpy(got[k])), as_bytes(ref[k])), k
    # groups of one map merge consistently; most groups with a foreign member do not
    bad_g = foreign.reshape(G, gs).any(axis=1)
    assert (ref["contra"][~bad_g] == 0).all()
    assert ref["contra"][bad_g].sum() >= 1
    assert (mask_ok == 1).all()
    merged.close()
    st.close()


def test_merge_rejects_bad_groups():
    dev = cuda_device()
    binding = lib()
    st = binding.Store(np.array([5, 5, 9], np.int32), device=dev)
    with pytest.raises(binding.F2Error) as e:  # widths differ within a group
        st.merge(np.array([0, 0, 0], np.int32), 1)
    assert e.value.code == 2
    with pytest.raises(binding.F2Error) as e:  # group id out of range
        st.merge(np.array([0, 1, 2], np.int32), 2)
    assert e.value.code == 3
    with pytest.raises(binding.F2Error) as e:  # an empty group
        st.merge(np.array([0, 0, -1], np.int32), 2)
    assert e.value.code == 1
    merged, ok = st.merge(np.array([0, 0, 1], np.int32), 2)  # empty bases merge to rank 0
    b = merged.basis()
    assert binding.to_numpy(b["rank"]).tolist() == [0, 0] and ok.tolist() == [1, 1]
    merged.close()
    st.close()


def test_shard_merge_equals_single_pass():
    """A context's stream learned as three shards and merged (Sec. 3: the
    retained rows of shards eliminated together) has the single-pass basis
    where the stream is consistent; the stream is inconsistent iff a shard or
    the merge flags a contradiction.  Checked against the GPU's own
    single-pass result (a property that needs no oracle) and the oracle."""
    dev = cuda_device()
    binding = lib()
    wl = wlmod.generate(wlmod.scaled(2, 300), 505)
    C = wl.num_ctx
    rng = np.random.default_rng(5)
    shard_rows, shard_bits = [], []
    for c in range(C):
        x, y = wl.ctx_rows(c)
        cut = np.sort(rng.integers(0, len(y) + 1, 2))
        for a, b in ((0, cut[0]), (cut[0], cut[1]), (cut[1], len(y))):
            shard_rows.append([(x[i], y[i]) for i in range(a, b)])
            shard_bits.append(wl.n_bits[c])
    from gpu_util import csr_from_rows

    ro, xo, x, y = csr_from_rows(np.array(shard_bits), shard_rows)
    whole = binding.Store(wl.n_bits, device=dev)
    gpu_learn_workload(binding, whole, wl, dev)
    shards = binding.Store(np.array(shard_bits, np.int32), device=dev)
    shards.learn(*(binding.to_device(a, dev) for a in (ro, x, xo, y)))
    merged, _ = shards.merge((np.arange(3 * C) // 3).astype(np.int32), C)
    W, S, M = whole.basis(), shards.basis(), merged.basis()
    torch.cuda.synchronize()
    W, S, M = ({k: binding.to_numpy(t[k]) for k in KEYS} for t in (W, S, M))
    single_contra = W["contra"] != 0
    either = (S["contra"].reshape(C, 3).any(axis=1)) | (M["contra"] != 0)
    assert np.array_equal(single_contra, either) and single_contra.any()
    ok = np.flatnonzero(~single_contra)
    for c in ok:
        sl = slice(int(whole.slot_off[c]), int(whole.slot_off[c + 1]))
        assert np.array_equal(W["basis_z"][sl], M["basis_z"][int(merged.slot_off[c]):int(merged.slot_off[c + 1])]), c
        sl = slice(int(whole.xw_off[c]), int(whole.xw_off[c + 1]))
        assert np.array_equal(W["basis_x"][sl], M["basis_x"][int(merged.xw_off[c]):int(merged.xw_off[c + 1])]), c
        sl = slice(int(whole.pw_off[c]), int(whole.pw_off[c + 1]))
        assert np.array_equal(W["pivot_mask"][sl], M["pivot_mask"][int(merged.pw_off[c]):int(merged.pw_off[c + 1])]), c
    assert np.array_equal(W["rank"][ok], M["rank"][ok])
    # the merge itself against the oracle's
    O = oracle.Oracle(np.array(shard_bits, np.int32), threads=4)
    O.learn(ro, xo, x, y)
    ex = O.export()
    d = np.array(shard_bits, np.int64) + 1
    grp = [[] for _ in range(C)]
    for s in range(3 * C):
        grp[s // 3] += _export_rows(ex, O.layout, s, int(d[s]))
    mro, mxo, mx, my = csr_from_rows(d[::3], grp)
    OM = oracle.Oracle(d[::3], raw=True, threads=4)
    OM.learn(mro, mxo, mx, my)
    ref = OM.export()
    for k in KEYS:
        assert np.array_equal(as_bytes(M[k]), as_bytes(ref[k])), k
    for s in (merged, shards, whole):
        s.close()
