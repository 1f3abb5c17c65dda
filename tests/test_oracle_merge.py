"""Map pooling in the oracle (Sec. 3): merged bases checked by enumeration.

The merged basis must span the union of the members' spans (|span| =
2^rank, checked by enumerating XORs of subsets), be the unique reduced
echelon form of it, and be consistent exactly when one linear map agrees
with every member on its span (checked by walking the union span and
carrying words: a vector reached with two different words is a conflict)."""
import random

import pytest

from oracle import f2_bigint as bi


def _span_words(rows):
    """{vector: word} over the span of (r, z) pairs, or None on a conflict."""
    span = {0: 0}
    for r, z in rows:
        new = {}
        for v, w in span.items():
            u, wu = v ^ r, w ^ z
            if u in span and span[u] != wu:
                return None
            if u in new and new[u] != wu:
                return None
            new[u] = wu
        span.update(new)
    return span


def _member(rng, d, M, dim):
    gens = [rng.getrandbits(d) for _ in range(dim)]
    rows = []
    for _ in range(rng.randint(1, 12)):
        v = 0
        for g in gens:
            if rng.random() < 0.5:
                v ^= g
        z = 0
        for j in range(d):
            if (v >> j) & 1:
                z ^= M[j]
        rows.append((v, z))
    return bi.learn_rows(d, rows)


@pytest.mark.parametrize("seed", range(30))
def test_merge_by_enumeration(seed):
    rng = random.Random(seed)
    d = rng.randint(2, 9)
    M = [rng.getrandbits(16) for _ in range(d)]
    members = [_member(rng, d, M, rng.randint(1, 4)) for _ in range(rng.randint(2, 4))]
    foreign = seed % 3 == 0
    if foreign:  # one member from another map
        M2 = [w ^ (rng.getrandbits(16) if rng.random() < 0.5 else 0) for w in M]
        members.append(_member(rng, d, M2, rng.randint(1, 4)))
    merged = bi.merge_bases(d, members)
    all_rows = [B.rows[k] for B in members for k in sorted(B.rows)]
    span = _span_words(all_rows)
    # union span size fixes the rank; the pivots and reduced rows are unique
    vecs = {0}
    for r, _ in all_rows:
        vecs |= {v ^ r for v in vecs}
    assert 2 ** merged.rank == len(vecs)
    assert sorted(merged.rows) == sorted({v.bit_length() - 1 for v in vecs if v})
    assert (span is None) == (merged.contradictions > 0)
    if span is not None:
        for k, (r, z) in merged.rows.items():
            assert span[r] == z
    if not foreign:
        assert merged.contradictions == 0


def test_merge_with_itself_is_idempotent():
    rng = random.Random(9)
    d = 8
    M = [rng.getrandbits(32) for _ in range(d)]
    B = _member(rng, d, M, 4)
    merged = bi.merge_bases(d, [B, B])
    assert merged.rows == B.rows and merged.contradictions == 0
