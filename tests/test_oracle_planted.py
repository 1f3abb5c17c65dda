"""Oracle checks on planted-map workloads (the four checks of the method's
acceptance criteria) plus structural invariants.

(a) a planted affine map is recovered exactly on full-rank contexts, and
    agrees with the planted one on the span otherwise;
(b) ranks match enumeration (see test_oracle_bruteforce.py);
(c) every injected contradiction is flagged, no clean context is, and the
    flag equals [rank([Phi|Y]) != rank(Phi)] (Sec. 2.3, consistency test)
    computed by a separate elimination over the full augmented rows;
(d) every training word is reproduced, planted out-of-span queries are
    rejected and in-span queries return the planted A x ^ b.
"""
import numpy as np
import pytest

import oracle
from oracle import f2_bigint as bi
from paper_2608_20532_gb300 import workloads as wlmod


def _planted_word(wl, c, xwords):
    n = int(wl.n_bits[c])
    a0 = int(wl.a_off[c])
    acc = wl.b[c].copy()
    for j in range(n):
        if (int(xwords[j // 32]) >> (j % 32)) & 1:
            acc ^= wl.A[a0 + j]
    return acc


def _learn(wl, threads=4):
    O = oracle.Oracle(wl.n_bits, threads=threads)
    O.learn_workload(wl)
    return O


@pytest.fixture(scope="module")
def cfg1():
    return wlmod.standard(1)


@pytest.fixture(scope="module")
def cfg1_oracle(cfg1):
    O = _learn(cfg1)
    return O, O.export()


def test_config1_contradictions(cfg1, cfg1_oracle):
    O, ex = cfg1_oracle
    injected = np.flatnonzero(cfg1.contra_pos >= 0)
    assert len(injected) == 3
    assert np.array_equal(np.flatnonzero(ex["contra"]), injected)
    assert np.array_equal(ex["first_contra"][injected], cfg1.contra_pos[injected])
    assert np.all(ex["n_contra"][injected] == 1)
    assert np.all(ex["first_contra"][ex["contra"] == 0] == -1)
    assert np.all(ex["rows_seen"] == cfg1.rows)


def test_config1_consistency_criterion(cfg1, cfg1_oracle):
    """flag == [rank([Phi|Y]) != rank(Phi)], ranks by a separate elimination."""
    O, ex = cfg1_oracle
    n = 48
    for c in range(cfg1.num_ctx):
        xs, ys = cfg1.ctx_rows(c)
        phis = [bi.phi(bi.words_to_int(xr), n) for xr in xs]
        aug = [p | (bi.words_to_int(yr) << (n + 1)) for p, yr in zip(phis, ys)]
        rphi, raug = bi.rank_of(phis), bi.rank_of(aug)
        assert ex["rank"][c] == rphi
        assert ex["contra"][c] == int(raug != rphi)


def test_config1_structure(cfg1, cfg1_oracle):
    """The one-hot modifier group ties its parity to the constant, so the
    constant column is never a pivot and rank <= 48 < d = 49."""
    O, ex = cfg1_oracle
    assert np.all(ex["rank"] <= 48)
    assert np.all(ex["pivot_mask"][0::2] & 1 == 0)
    assert np.all(ex["rank"] >= 40)


def test_config1_encode(cfg1, cfg1_oracle):
    O, ex = cfg1_oracle
    q = cfg1.queries
    y, ok = O.encode(q.ctx_id, q.x)
    assert np.array_equal(ok, q.expect_in)  # planted out-of-span queries are rejected
    assert not y[ok == 0].any()
    for i in np.flatnonzero(ok)[:1500]:
        assert np.array_equal(y[i], _planted_word(cfg1, int(q.ctx_id[i]), q.x[i]))
    # every training word is reproduced (all rows but the injected ones)
    for c in range(0, cfg1.num_ctx, 7):
        xs, ys = cfg1.ctx_rows(c)
        yy, okk = O.encode(np.full(len(xs), c, np.int32), xs)
        assert okk.all()
        keep = np.ones(len(xs), bool)
        if cfg1.contra_pos[c] >= 0:
            keep[cfg1.contra_pos[c]] = False
        assert np.array_equal(yy[keep], ys[keep])


def test_config1_solve_on_span(cfg1, cfg1_oracle):
    """Rank-deficient contexts: the solved (A', b') agrees with the planted map
    on every training x (free coordinates are zero, Sec. 2.3)."""
    O, ex = cfg1_oracle
    W = O.solve()
    L = O.layout
    for c in range(0, cfg1.num_ctx, 5):
        s0 = int(L["slot_off"][c])
        xs, ys = cfg1.ctx_rows(c)
        for i in range(0, len(xs), 13):
            if i == cfg1.contra_pos[c]:
                continue
            acc = W[s0].copy()
            for j in range(48):
                if (int(xs[i][j // 32]) >> (j % 32)) & 1:
                    acc ^= W[s0 + 1 + j]
            assert np.array_equal(acc, ys[i])


def _full_rank_workload(num_ctx=24, n=40, rows=160, seed=77):
    cfg = dict(num_ctx=num_ctx, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=n, rows_fixed=rows,
               dup_frac=0.0, density=0.5, n_contra=3)
    return wlmod.generate(cfg, seed)


def test_planted_map_recovered_exactly():
    """Check (a): uniform features give rank d, and then (A, b) is the planted map."""
    wl = _full_rank_workload()
    O = _learn(wl)
    ex = O.export()
    assert np.all(ex["rank"] == 41)
    W = O.solve()
    for c in range(wl.num_ctx):
        s0 = int(O.layout["slot_off"][c])
        assert np.array_equal(W[s0], wl.b[c])
        a0 = int(wl.a_off[c])
        assert np.array_equal(W[s0 + 1:s0 + 41], wl.A[a0:a0 + 40])
    injected = np.flatnonzero(wl.contra_pos >= 0)
    assert np.array_equal(np.flatnonzero(ex["contra"]), injected)
    assert np.array_equal(ex["first_contra"][injected], wl.contra_pos[injected])


def _views(O):
    ex = O.export()
    return [oracle.ctx_view(ex, O.layout, c) for c in range(O.num_ctx)]


def test_rref_and_pair_invariant(cfg1, cfg1_oracle):
    """Reduced form (each pivot column is set only in its own row, the pivot is
    the row's highest bit) and r_k W = z_k (Appendix C, basis-pair invariant)."""
    O, ex = cfg1_oracle
    W = O.solve()
    for c in range(0, cfg1.num_ctx, 3):
        v = oracle.ctx_view(ex, O.layout, c)
        s0 = int(O.layout["slot_off"][c])
        pm = bi.words_to_int(v["pivot_mask"])
        for k in range(v["d"]):
            r = bi.words_to_int(v["basis_x"][k])
            if not (pm >> k) & 1:
                assert r == 0
                continue
            assert r.bit_length() - 1 == k
            assert (r & pm) == (1 << k)
            acc = 0
            for j in range(v["d"]):
                if (r >> j) & 1:
                    acc ^= bi.words_to_int(W[s0 + j])
            assert acc == bi.words_to_int(v["basis_z"][k])


def _subset_workload(wl, ctxs, perm_seed=None, split=None):
    """Rows of the chosen contexts, optionally permuted, as a CSR batch."""
    rng = np.random.default_rng(perm_seed)
    nb, xs, ys, rows = [], [], [], []
    for c in ctxs:
        x, y = wl.ctx_rows(c)
        idx = np.arange(len(x))
        if perm_seed is not None:
            idx = rng.permutation(len(x))
        nb.append(int(wl.n_bits[c]))
        xs.append(x[idx].reshape(-1))
        ys.append(y[idx])
        rows.append(len(x))
    row_off = np.zeros(len(ctxs) + 1, np.int64)
    row_off[1:] = np.cumsum(rows)
    W = [(n + 31) // 32 for n in nb]
    x_off = np.zeros(len(ctxs), np.int64)
    x_off[1:] = np.cumsum([r * w for r, w in zip(rows, W)])[:-1]
    return np.array(nb, np.int32), row_off, x_off, np.concatenate(xs), np.concatenate(ys)


def test_permutation_invariance_on_consistent_contexts():
    wl = wlmod.generate(wlmod.scaled(2, 48), 11)
    clean = [c for c in range(wl.num_ctx) if wl.contra_pos[c] < 0][:30]
    nb, ro, xo, x, y = _subset_workload(wl, clean)
    O1 = oracle.Oracle(nb, threads=2)
    O1.learn(ro, xo, x, y)
    nb2, ro2, xo2, x2, y2 = _subset_workload(wl, clean, perm_seed=5)
    O2 = oracle.Oracle(nb2, threads=2)
    O2.learn(ro2, xo2, x2, y2)
    e1, e2 = O1.export(), O2.export()
    for k in ("rank", "pivot_mask", "basis_x", "basis_z", "contra"):
        assert np.array_equal(e1[k], e2[k]), k


def test_incremental_batches_equal_single_pass():
    wl = wlmod.generate(wlmod.scaled(2, 40), 12)
    O1 = _learn(wl)
    O2 = oracle.Oracle(wl.n_bits, threads=3)
    # three incremental calls: rows [0, t/3), [t/3, 2t/3), [2t/3, t) of every context
    for part in range(3):
        lo = wl.row_off[:-1] + (wl.rows * part) // 3
        hi = wl.row_off[:-1] + (wl.rows * (part + 1)) // 3
        cnt = hi - lo
        ro = np.zeros(wl.num_ctx + 1, np.int64)
        ro[1:] = np.cumsum(cnt)
        Wc = (wl.n_bits.astype(np.int64) + 31) // 32
        xs = np.concatenate([wl.x[wl.x_off[c] + (lo[c] - wl.row_off[c]) * Wc[c]:
                                  wl.x_off[c] + (hi[c] - wl.row_off[c]) * Wc[c]] for c in range(wl.num_ctx)])
        xo = np.zeros(wl.num_ctx, np.int64)
        xo[1:] = np.cumsum(cnt * Wc)[:-1]
        ys = np.concatenate([wl.y[lo[c]:hi[c]] for c in range(wl.num_ctx)])
        O2.learn(ro, xo, xs, ys)
    e1, e2 = O1.export(), O2.export()
    for k in e1:
        assert np.array_equal(e1[k], e2[k]), k


def test_shard_merge_reproduces_span():
    """Bases of two shards merged by eliminating their retained rows give the
    basis of the whole stream (Sec. 2.2, mergeable bases), for consistent contexts."""
    wl = wlmod.generate(wlmod.scaled(2, 24), 13)
    for c in [c for c in range(wl.num_ctx) if wl.contra_pos[c] < 0][:8]:
        xs, ys = wl.ctx_rows(c)
        n = int(wl.n_bits[c])
        rows = [(bi.phi(bi.words_to_int(xr), n), bi.words_to_int(yr)) for xr, yr in zip(xs, ys)]
        h = len(rows) // 2
        whole = bi.learn_rows(n + 1, rows)
        a = bi.learn_rows(n + 1, rows[:h])
        b = bi.learn_rows(n + 1, rows[h:])
        merged = bi.learn_rows(n + 1, list(b.rows.values()) + list(a.rows.values()))
        assert merged.rows == whole.rows
        assert merged.contradictions == 0


def test_c_and_bigint_oracles_agree():
    wl = wlmod.generate(wlmod.scaled(2, 40), 14)
    O = _learn(wl)
    ex = O.export()
    for c in range(wl.num_ctx):
        xs, ys = wl.ctx_rows(c)
        n = int(wl.n_bits[c])
        B = bi.learn_rows(n + 1, [(bi.phi(bi.words_to_int(xr), n), bi.words_to_int(yr))
                                  for xr, yr in zip(xs, ys)])
        v = oracle.ctx_view(ex, O.layout, c)
        got = {k: (bi.words_to_int(v["basis_x"][k]), bi.words_to_int(v["basis_z"][k]))
               for k in range(v["d"]) if (int(v["pivot_mask"][k // 32]) >> (k % 32)) & 1}
        assert got == B.rows
        assert v["n_contra"] == B.contradictions
        assert v["first_contra"] == (B.first_contradiction if B.first_contradiction is not None else -1)


def test_threads_do_not_change_results():
    wl = wlmod.generate(wlmod.scaled(3, 60), 15)
    e1 = _learn(wl, threads=1).export()
    e8 = _learn(wl, threads=8).export()
    for k in e1:
        assert np.array_equal(e1[k], e8[k]), k
    assert e1["contra"].sum() == 0  # no contradictions injected in config 3
