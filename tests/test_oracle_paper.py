"""Pins of the CPU oracle against the paper's worked examples.

Appendix B (streaming elimination trace), Appendix C (HMMA feature vector,
Table 6 basis pairs, learned word, scheduler-control merge, little-endian
bytes) and Appendix D (128-bit numbering of bits 122 and 124).  Fixtures live
in tests/golden/ with their citations.
"""
import json
import os

import numpy as np

import oracle
from oracle import f2_bigint as bi


def _load(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


def _b(s):
    return int(s, 2)


# --------------------------------------------------------------- Appendix B

def test_appendix_b_bigint_trace(golden_dir):
    g = _load(golden_dir, "appendix_b_trace.json")
    B = bi.Basis(g["d"])
    got = []
    for i, (q, y) in enumerate(g["observations"]):
        got.append(B.learn(_b(q), _b(y)))
        if i == 0:
            assert B.rows == {int(k): (_b(r), _b(z)) for k, (r, z) in g["after_observation_1"].items()}
        if i == 1:
            assert B.rows == {int(k): (_b(r), _b(z)) for k, (r, z) in g["after_observation_2"].items()}
            kind, _, visited, r, z = B.trace[-1]
            assert (r, z) == tuple(_b(v) for v in g["reduction_of_observation_2"]["residual"])
            assert r.bit_length() - 1 == g["reduction_of_observation_2"]["pivot"]
        if i == 2:
            kind, _, visited, r, z = B.trace[-1]
            assert (r, z) == tuple(_b(v) for v in g["reduction_of_observation_3"]["residual"])
            assert r.bit_length() - 1 == g["reduction_of_observation_3"]["pivot"]
    assert got == g["classification"]
    assert B.trace[3][2] == g["observation_4_visits"]
    assert B.rows == {int(k): (_b(r), _b(z)) for k, (r, z) in g["final_basis"].items()}
    assert B.rank == 3

    # encode trace of the supported query: residual and accumulator after each pivot
    enc = g["encode_supported"]
    q, acc = _b(enc["query"]), 0
    steps = [(q, acc)]
    for k in enc["visits"]:
        rk, zk = B.rows[k]
        assert (q >> k) & 1
        q, acc = q ^ rk, acc ^ zk
        steps.append((q, acc))
    assert steps == [(_b(a), _b(b)) for a, b in enc["trace"]]
    assert B.encode(_b(enc["query"])) == (True, _b(enc["word"]), 0)
    rej = g["encode_rejected"]
    ok, word, res = B.encode(_b(rej["query"]))
    assert (ok, word, res) == (False, 0, _b(rej["residual"]))

    # contradiction variant
    C = bi.Basis(g["d"])
    obs = list(g["observations"])
    obs[3] = [obs[3][0], g["contradiction_variant"]["observation_4_word"]]
    kinds = [C.learn(_b(q), _b(y)) for q, y in obs]
    assert kinds == ["new", "new", "new", "contradiction"]
    _, idx, _, r, z = C.trace[-1]
    assert (r, z) == tuple(_b(v) for v in g["contradiction_variant"]["residual"])
    assert C.contradictions == 1 and C.first_contradiction == 3
    assert C.rows == B.rows  # the contradicting row is not inserted


def _c_oracle_rows(g, obs):
    """Feed Appendix B rows one at a time through the C oracle (raw feature rows)."""
    O = oracle.Oracle([g["d"]], raw=True, threads=1)
    snaps = []
    for q, y in obs:
        x = np.array([_b(q)], np.uint32)
        yy = np.array([[_b(y), 0, 0, 0]], np.uint32)
        O.learn(np.array([0, 1], np.int64), np.array([0], np.int64), x, yy)
        snaps.append(oracle.ctx_view(O.export(), O.layout, 0))
    return O, snaps


def _basis_dict(view):
    out = {}
    for k in range(view["d"]):
        if (int(view["pivot_mask"][k // 32]) >> (k % 32)) & 1:
            out[k] = (int(view["basis_x"][k][0]), int(view["basis_z"][k][0]))
        else:
            assert not view["basis_x"][k].any() and not view["basis_z"][k].any()
    return out


def test_appendix_b_c_oracle(golden_dir):
    g = _load(golden_dir, "appendix_b_trace.json")
    O, snaps = _c_oracle_rows(g, g["observations"])
    assert _basis_dict(snaps[0]) == {int(k): (_b(r), _b(z)) for k, (r, z) in g["after_observation_1"].items()}
    assert _basis_dict(snaps[1]) == {int(k): (_b(r), _b(z)) for k, (r, z) in g["after_observation_2"].items()}
    assert [s["rank"] for s in snaps] == [1, 2, 3, 3]
    final = _basis_dict(snaps[-1])
    assert final == {int(k): (_b(r), _b(z)) for k, (r, z) in g["final_basis"].items()}
    assert snaps[-1]["contra"] == 0 and snaps[-1]["n_contra"] == 0 and snaps[-1]["first_contra"] == -1
    assert snaps[-1]["rows_seen"] == 4

    q = np.array([[_b(g["encode_supported"]["query"])], [_b(g["encode_rejected"]["query"])]], np.uint32)
    y, ok = O.encode(np.zeros(2, np.int32), q)
    assert ok.tolist() == [1, 0]
    assert int(y[0][0]) == _b(g["encode_supported"]["word"]) and not y[0][1:].any()
    assert not y[1].any()

    W = O.solve()
    # W[k] = z_k on the pivots 3, 2, 1 and zero on the free coordinate 0
    assert [int(w[0]) for w in W] == [0, final[1][1], final[2][1], final[3][1]]

    obs = list(g["observations"])
    obs[3] = [obs[3][0], g["contradiction_variant"]["observation_4_word"]]
    _, snaps2 = _c_oracle_rows(g, obs)
    s = snaps2[-1]
    assert (s["contra"], s["first_contra"], s["n_contra"], s["rank"]) == (1, 3, 1, 3)
    assert _basis_dict(s) == final


# --------------------------------------------------------------- Appendix C

def _hex128(s):
    return int(s, 16)


def _feature_index(f):
    return 0 if f == "const" else 1 + 64 * f[0] + f[1]


def test_appendix_c_feature_vector(golden_dir):
    g = _load(golden_dir, "appendix_c_hmma.json")
    f = bi.parsed_value_features(g["values"])
    active = [k for k in range(g["feature_width"]) if (f >> k) & 1]
    assert active == [0, 1, 2, 3, 67, 131, 135, 196, 199, 259]
    assert f.bit_length() <= g["feature_width"]
    rows = {r["k"]: sum(1 << _feature_index(t) for t in r["features"]) for r in g["basis_rows"]}
    # Eq. hmma-feature-reduction: phi(x) = r_259 ^ r_199 ^ r_196 ^ r_135 ^ r_3
    acc = 0
    for k, r in rows.items():
        assert r.bit_length() - 1 == k  # pivot = highest active feature
        acc ^= r
    assert acc == f


def test_appendix_c_encode(golden_dir):
    g = _load(golden_dir, "appendix_c_hmma.json")
    d = g["feature_width"]
    rows = [(sum(1 << _feature_index(t) for t in r["features"]), _hex128(r["z"])) for r in g["basis_rows"]]
    f = bi.parsed_value_features(g["values"])
    want = _hex128(g["y_learned"])

    B = bi.learn_rows(d, rows)
    assert B.rank == 5 and sorted(B.rows) == [3, 135, 196, 199, 259]
    assert B.encode(f) == (True, want, 0)

    # the same through the C oracle (raw feature rows of width 321)
    nw = (d + 31) // 32
    x = np.array([bi.int_to_words(r, nw) for r, _ in rows], np.uint32).reshape(-1)
    y = np.array([bi.int_to_words(z, 4) for _, z in rows], np.uint32)
    O = oracle.Oracle([d], raw=True, threads=1)
    O.learn(np.array([0, 5], np.int64), np.array([0], np.int64), x, y)
    v = oracle.ctx_view(O.export(), O.layout, 0)
    assert v["rank"] == 5
    yq, ok = O.encode(np.zeros(1, np.int32), np.array([bi.int_to_words(f, nw)], np.uint32))
    assert ok.tolist() == [1]
    assert bi.words_to_int(yq[0]) == want
    # flipping the constant of the query leaves the span (no stored row supplies it alone)
    _, ok2 = O.encode(np.zeros(1, np.int32), np.array([bi.int_to_words(f ^ 1, nw)], np.uint32))
    assert ok2.tolist() == [0]


def test_appendix_c_word_numbering(golden_dir):
    """Scheduler-control merge and little-endian emission fix the 128-bit numbering."""
    g = _load(golden_dir, "appendix_c_hmma.json")
    y_learned = _hex128(g["y_learned"])
    sc = int(g["sched_control"], 16)
    shifted = sc << g["sched_shift"]
    assert shifted == _hex128(g["sched_shifted"])
    assert sc < (1 << 17)  # 17 control bits at 105..121
    y_full = y_learned ^ shifted
    assert y_full == _hex128(g["y_full"])
    words = np.array(bi.int_to_words(y_full, 4), np.uint32)
    le = words.astype("<u4").tobytes()
    assert le.hex(" ") == g["le_bytes"]


# --------------------------------------------------------------- Appendix D

def test_appendix_d_bits(golden_dir):
    g = _load(golden_dir, "appendix_d_depbar.json")
    a, b = _hex128(g["word_a"]), _hex128(g["word_b"])
    assert a ^ b == _hex128(g["xor"])
    wa = np.array(bi.int_to_words(a, 4), np.uint32)
    wb = np.array(bi.int_to_words(b, 4), np.uint32)
    x = wa ^ wb
    bits = [i for i in range(128) if (int(x[i // 32]) >> (i % 32)) & 1]
    assert bits == g["xor_bits"]


# ------------------------------------------------------- encode epilogue

def test_epilogue_appendix_c(golden_dir):
    """Eq. hmma-full-word: the learned word XOR (sc << 105), emitted as the
    16 little-endian bytes the paper prints."""
    g = _load(golden_dir, "appendix_c_hmma.json")
    y_learned = _hex128(g["y_learned"])
    full = bi.encode_epilogue(y_learned, True, sched=int(g["sched_control"], 16))
    assert full == _hex128(g["y_full"])
    le = np.array(bi.int_to_words(full, 4), np.uint32).astype("<u4").tobytes()
    assert le.hex(" ") == g["le_bytes"]
    assert bi.encode_epilogue(y_learned, False, sched=int(g["sched_control"], 16)) == 0  # rejected: no word


def test_epilogue_appendix_d(golden_dir):
    """Appendix D: words A and B differ only in the opaque bits 122 and 124;
    restoring them from the recorded state gives back either word."""
    g = _load(golden_dir, "appendix_d_depbar.json")
    a, b = _hex128(g["word_a"]), _hex128(g["word_b"])
    mask = sum(1 << k for k in g["xor_bits"])
    learned = a & ~mask  # the learned map excludes the masked bits
    assert learned == b & ~mask
    assert bi.encode_epilogue(learned, True, state=b, mask=mask) == b
    assert bi.encode_epilogue(learned, True, state=a, mask=mask) == a
    assert bi.encode_epilogue(a, True) == a  # no control, no mask: unchanged
    # only the 17 control bits are merged, at 105..121, below the opaque bits
    assert bi.encode_epilogue(0, True, sched=(1 << 17) | 1) == 1 << 105
    assert bi.encode_epilogue(0, True, sched=(1 << 17) - 1) == ((1 << 17) - 1) << 105
    assert ((((1 << 17) - 1) << 105) & mask) == 0
