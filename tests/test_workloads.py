"""Properties of the seeded workload generator (input synthesis only)."""
import numpy as np

from paper_2608_20532_gb300 import workloads as wlmod


def _bits(words, j):
    return (int(words[j // 32]) >> (j % 32)) & 1


def test_config1_shape():
    wl = wlmod.standard(1)
    assert wl.num_ctx == 256 and np.all(wl.n_bits == 48)
    assert np.all(wl.rows == 260) and wl.total_rows == 66560
    assert wl.queries.x.shape == (25600, 2)
    assert (wl.contra_pos >= 0).sum() == 3
    assert abs(wl.queries.expect_in.mean() - 0.5) < 0.03


def test_rows_follow_planted_map_and_layout():
    wl = wlmod.generate(wlmod.scaled(2, 64), 3)
    go = wlmod.onehot_offset(wl.params["layout"])
    for c in range(wl.num_ctx):
        xs, ys = wl.ctx_rows(c)
        n = int(wl.n_bits[c])
        W = (n + 31) // 32
        assert xs.shape == (wl.rows[c], W)
        if n % 32:
            assert not (xs[:, -1] >> np.uint32(n % 32)).any()  # bits >= n are zero
        onehot = sum(((xs[:, (go + t) // 32] >> np.uint32((go + t) % 32)) & 1) for t in range(8))
        assert np.all(onehot == 1)
        a0 = int(wl.a_off[c])
        for i in range(0, len(xs), 17):
            acc = wl.b[c].copy()
            for j in range(n):
                if _bits(xs[i], j):
                    acc ^= wl.A[a0 + j]
            flips = int(np.unpackbits((acc ^ ys[i]).view(np.uint8)).sum())
            assert flips == (1 if i == wl.contra_pos[c] else 0)


def test_contradiction_is_flipped_copy_of_earlier_row():
    wl = wlmod.generate(wlmod.scaled(2, 400), 4)
    for c in np.flatnonzero(wl.contra_pos >= 0):
        xs, ys = wl.ctx_rows(c)
        p = int(wl.contra_pos[c])
        same = [i for i in range(p) if np.array_equal(xs[i], xs[p])]
        assert same
        diff = ys[same[0]] ^ ys[p]
        assert int(np.unpackbits(diff.view(np.uint8)).sum()) == 1
        bit = int(wl.contra_bit[c])
        assert (int(diff[bit // 32]) >> (bit % 32)) & 1


def test_deterministic_and_thread_independent():
    a = wlmod.generate(wlmod.scaled(3, 50), 9, nthreads=1)
    b = wlmod.generate(wlmod.scaled(3, 50), 9, nthreads=7)
    for k in ("n_bits", "rows", "x", "y", "A", "b", "contra_pos", "two_stream"):
        assert np.array_equal(getattr(a, k), getattr(b, k)), k
    assert np.array_equal(a.queries.x, b.queries.x) and np.array_equal(a.queries.ctx_id, b.queries.ctx_id)
    c = wlmod.generate(wlmod.scaled(3, 50), 10, nthreads=3)
    assert not np.array_equal(a.y[:100], c.y[:100])


def test_batch_major_layout():
    cfg = dict(num_ctx=3, layout=wlmod.LAYOUT_UNIFORM_BITS, n_fixed=70, rows_fixed=40, dup_frac=0.0,
               density=0.5, n_contra=1, batch_rows=10)
    wl = wlmod.generate(cfg, 5)
    assert len(wl.batches) == 4
    ro, xo = wl.batches[2]
    assert ro[0] == 2 * 3 * 10 and np.all(np.diff(ro) == 10)
    x, y = wl.ctx_rows(1)
    assert x.shape == (40, 3) and y.shape == (40, 4)
    assert np.array_equal(y[20:30], wl.y[ro[1]:ro[2]])


def test_zipf_queries():
    wl = wlmod.generate(wlmod.scaled(3, 300), 21, query_count=20000)
    q = wl.queries
    counts = np.bincount(q.ctx_id, minlength=wl.num_ctx)
    top = np.sort(counts)[::-1]
    assert top[0] > 10 * np.median(counts[counts > 0])  # heavy head
    assert abs((1 - q.expect_in.mean()) - 0.05) < 0.01


def test_parsed_lowrank_layout_and_map():
    """Parsed-value rows: x is the k int64 values' little-endian memory
    (feature bit 64i + b = bit b of v_i, Sec. 2.1); y follows the planted
    affine map except the one flipped duplicate of a contradiction context."""
    wl = wlmod.parsed_lowrank(num_ctx=60, seed=3, rows_per_rank=20)
    assert (wl.n_bits % 64 == 0).all() and wl.n_bits.min() >= 128 and wl.n_bits.max() <= 512
    for c in range(wl.num_ctx):
        xs, ys = wl.ctx_rows(c)
        k = int(wl.n_bits[c]) // 64
        vals = np.ascontiguousarray(xs).view(np.int64)
        assert vals.shape == (int(wl.rows[c]), k)
        n = int(wl.n_bits[c])
        a0 = int(wl.a_off[c])
        for i in range(0, len(xs), 7):
            acc = wl.b[c].copy()
            for j in range(n):
                if (int(vals[i, j // 64]) >> (j % 64)) & 1:
                    acc ^= wl.A[a0 + j]
            flips = int(np.unpackbits((acc ^ ys[i]).view(np.uint8)).sum())
            assert flips == (1 if i == wl.contra_pos[c] else 0)
        # at most 2^(r-1) distinct x (an affine subspace of dimension r - 1)
        assert len({bytes(r) for r in xs}) <= 2 ** (int(wl.fresh[c]) - 1)


def test_parsed_lowrank_groups_share_the_map():
    """Consecutive contexts in groups of group_size share k and the planted
    (A, b) (the exact contexts of one (f, m) group); different groups draw
    their own."""
    gs = 4
    wl = wlmod.parsed_lowrank(num_ctx=24, seed=5, rows_per_rank=10, group_size=gs)
    for g0 in range(0, wl.num_ctx, gs):
        n = int(wl.n_bits[g0])
        a0 = int(wl.a_off[g0])
        for c in range(g0, g0 + gs):
            assert int(wl.n_bits[c]) == n
            ac = int(wl.a_off[c])
            assert np.array_equal(wl.A[ac:ac + n], wl.A[a0:a0 + n])
            assert np.array_equal(wl.b[c], wl.b[g0])
    firsts = list(range(0, wl.num_ctx, gs))
    maps = {(int(wl.n_bits[c]), bytes(wl.b[c])) for c in firsts}
    assert len(maps) == len(firsts)
