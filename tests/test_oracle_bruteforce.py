"""Brute-force pins of the oracle on tiny systems.

For random k x d systems (k <= 16 rows, d <= 12 feature bits) every quantity
the oracle reports is recomputed by enumeration, without elimination:

* the span S = {XOR of subsets of rows}: |S| = 2^rank;
* the pivot set = {msb(v) : v in S, v != 0};
* the reduced basis row of pivot p = the unique v in S with msb p that is
  zero at every other pivot position (the reduced echelon form is unique);
* the sequential contradiction semantics (Sec. 2.2 steps (2)-(3)): a row is a
  contradiction iff its features lie in the span of the rows accepted before
  it and its word differs from the word the accepted rows assign to them;
* encode (Sec. 2.3): accepted iff q in S, and then the word of q.
"""
import random

import numpy as np
import pytest

import oracle
from oracle import f2_bigint as bi


def _enumerate_accepted(rows):
    """Sequential semantics by enumeration: returns (span_map, kinds)."""
    span = {0: 0}
    kinds = []
    for r, z in rows:
        if r in span:
            kinds.append("redundant" if span[r] == z else "contradiction")
        else:
            span.update({v ^ r: w ^ z for v, w in list(span.items())})
            kinds.append("new")
    return span, kinds


def _rref_by_enumeration(span, d):
    nonzero = [v for v in span if v]
    pivots = sorted({v.bit_length() - 1 for v in nonzero})
    pmask = sum(1 << p for p in pivots)
    basis = {}
    for p in pivots:
        cands = [v for v in nonzero if v.bit_length() - 1 == p and (v & pmask) == (1 << p)]
        assert len(cands) == 1
        basis[p] = (cands[0], span[cands[0]])
    return pivots, basis


def _random_system(rng, k, d, consistent, dup_rate=0.3):
    rows = []
    M = [rng.getrandbits(16) for _ in range(d)]  # a linear map: feature bit j -> word M[j]
    for i in range(k):
        if rows and rng.random() < dup_rate:
            r = rows[rng.randrange(len(rows))][0]
            if rng.random() < 0.5:  # an XOR of two earlier rows
                r ^= rows[rng.randrange(len(rows))][0]
        else:
            r = rng.getrandbits(d)
        z = 0
        for j in range(d):
            if (r >> j) & 1:
                z ^= M[j]
        if not consistent and rng.random() < 0.25:
            z ^= 1 << rng.randrange(16)
        rows.append((r, z))
    return rows, M


@pytest.mark.parametrize("seed", range(40))
def test_bigint_matches_enumeration(seed):
    rng = random.Random(seed)
    d = rng.randint(1, 12)
    k = rng.randint(0, 16)
    rows, _ = _random_system(rng, k, d, consistent=(seed % 2 == 0))
    span, kinds = _enumerate_accepted(rows)
    B = bi.learn_rows(d, rows)
    assert [t[0] for t in B.trace] == kinds
    assert 2 ** B.rank == len(span)
    pivots, basis = _rref_by_enumeration(span, d)
    assert sorted(B.rows) == pivots
    assert B.rows == basis
    assert B.contradictions == kinds.count("contradiction")
    first = kinds.index("contradiction") if "contradiction" in kinds else None
    assert B.first_contradiction == first
    for q in range(1 << d):
        ok, word, res = B.encode(q)
        assert ok == (q in span)
        assert word == (span[q] if ok else 0)
        if not ok:
            assert res != 0 and not any((res >> p) & 1 for p in pivots)


def _words(v, n):
    return bi.int_to_words(v, (n + 31) // 32)


@pytest.mark.parametrize("seed", range(24))
def test_c_oracle_matches_enumeration(seed):
    """C oracle, raw feature rows, many tiny contexts in one store."""
    rng = random.Random(1000 + seed)
    C = 6
    ds, systems = [], []
    for c in range(C):
        d = rng.randint(1, 12)
        rows, _ = _random_system(rng, rng.randint(0, 16), d, consistent=(c % 2 == 0))
        ds.append(d)
        systems.append(rows)
    row_off = np.zeros(C + 1, np.int64)
    row_off[1:] = np.cumsum([len(s) for s in systems])
    x_off = np.zeros(C, np.int64)
    x_list, y_list, pos = [], [], 0
    for c, rows in enumerate(systems):
        x_off[c] = pos
        for r, z in rows:
            x_list.extend(_words(r, ds[c]))
            y_list.append(bi.int_to_words(z, 4))
            pos += (ds[c] + 31) // 32
    x = np.array(x_list, np.uint32)
    y = np.array(y_list, np.uint32).reshape(-1, 4)
    O = oracle.Oracle(ds, raw=True, threads=2)
    O.learn(row_off, x_off, x, y)
    ex = O.export()
    W = O.solve()
    for c, rows in enumerate(systems):
        v = oracle.ctx_view(ex, O.layout, c)
        span, kinds = _enumerate_accepted(rows)
        pivots, basis = _rref_by_enumeration(span, ds[c])
        assert v["rank"] == len(pivots) and 2 ** v["rank"] == len(span)
        got = {}
        for k in range(ds[c]):
            if (int(v["pivot_mask"][k // 32]) >> (k % 32)) & 1:
                got[k] = (bi.words_to_int(v["basis_x"][k]), bi.words_to_int(v["basis_z"][k]))
        assert got == basis
        nc = kinds.count("contradiction")
        assert v["n_contra"] == nc and v["contra"] == int(nc > 0)
        assert v["first_contra"] == (kinds.index("contradiction") if nc else -1)
        assert v["rows_seen"] == len(rows)
        s0 = int(O.layout["slot_off"][c])
        for k in range(ds[c]):
            wk = bi.words_to_int(W[s0 + k])
            assert wk == (basis[k][1] if k in basis else 0)
        # encode every vector of the feature space
        qs = list(range(1 << ds[c]))
        qx = np.array([_words(q, ds[c]) for q in qs], np.uint32)
        yq, ok = O.encode(np.full(len(qs), c, np.int32), qx)
        for i, q in enumerate(qs):
            assert ok[i] == int(q in span)
            assert bi.words_to_int(yq[i]) == (span[q] if q in span else 0)


def test_invalid_context_id_rejected():
    O = oracle.Oracle([5, 7], raw=False, threads=1)
    y, ok = O.encode(np.array([-1, 2, 0], np.int32), np.zeros((3, 1), np.uint32))
    assert ok.tolist() == [0xFF, 0xFF, 0]  # context 0 is empty: only q = 0 would be in span
    assert not y.any()


def test_invalid_widths():
    with pytest.raises(ValueError):
        oracle.Oracle([0])
    with pytest.raises(ValueError):
        oracle.Oracle([1025])
    oracle.Oracle([1024])  # d = 1025 is the largest supported row


def test_affine_phi_rows_and_constant_column():
    """Non-raw mode adds the constant at index 0: phi(x) = [1 || x] (Sec. 2.1)."""
    rng = random.Random(5)
    n = 9
    xs = [rng.getrandbits(n) for _ in range(30)]
    A = [rng.getrandbits(128) for _ in range(n)]
    b = rng.getrandbits(128)

    def f(x):
        y = b
        for j in range(n):
            if (x >> j) & 1:
                y ^= A[j]
        return y

    x = np.array([_words(v, n) for v in xs], np.uint32).reshape(-1)
    y = np.array([bi.int_to_words(f(v), 4) for v in xs], np.uint32)
    O = oracle.Oracle([n], threads=1)
    O.learn(np.array([0, len(xs)], np.int64), np.array([0], np.int64), x, y)
    B = bi.learn_rows(n + 1, [(bi.phi(v, n), f(v)) for v in xs])
    v = oracle.ctx_view(O.export(), O.layout, 0)
    got = {k: (bi.words_to_int(v["basis_x"][k]), bi.words_to_int(v["basis_z"][k]))
           for k in range(n + 1) if (int(v["pivot_mask"][k // 32]) >> (k % 32)) & 1}
    assert got == B.rows
    # with 30 random rows of 10 affine features the system is full rank, so the
    # solve returns the planted map exactly: W[0] = b, W[1+j] = column j of A
    assert v["rank"] == n + 1
    W = O.solve()
    assert bi.words_to_int(W[0]) == b
    assert [bi.words_to_int(W[1 + j]) for j in range(n)] == A
