"""Pins for the oracle's retrieval and candidate selection (Section 3.3).

The oracle's window comparison is checked against a substring search over an
encoded buffer (exhaustively on every short buffer over a 3-letter alphabet),
against hand-worked selections (tests/golden/select_cases.json) and against
the planted repeats of the synthetic workloads.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle
import synth


def _scan1(tokens, k, scores, theta, top_c, span_len, pos_cap=64, gate_ok=None):
    tokens = np.asarray(tokens, np.int32)
    return oracle.match_scan(tokens, np.array([0, tokens.size]), np.array([k]),
                             np.asarray(scores, np.float32), theta, top_c, span_len, pos_cap,
                             gate_ok=gate_ok)


def _find_all(X, k):
    """Ends of every earlier occurrence of the last k tokens, via str.find."""
    t = len(X)
    if k < 1 or k > t:
        return []
    s = "".join(chr(65 + x) for x in X)
    key = s[t - k:]
    hay = s[:t - 1]          # an occurrence must end at p <= t-2
    out, start = [], 0
    while True:
        j = hay.find(key, start)
        if j < 0:
            return out
        out.append(j + k - 1)
        start = j + 1        # overlapping occurrences too


def test_select_golden(golden_dir):
    cases = json.load(open(os.path.join(golden_dir, "select_cases.json")))["cases"]
    for c in cases:
        o = _scan1(c["tokens"], c["k"], c["scores"], c["theta_score"], c["top_c"], c["span_len"])
        assert o["count"][0] == c["count"], c["name"]
        assert o["pos"][0][:c["count"]].tolist() == c["pos"], c["name"]
        assert o["sel_pos"][0].tolist() == c["sel_pos"], c["name"]
        assert o["sel_len"][0].tolist() == c["sel_len"], c["name"]
        assert o["spans"][0].tolist() == c["spans"], c["name"]
        assert o["n_sel"][0] == sum(p >= 0 for p in c["sel_pos"]), c["name"]


def test_exhaustive_short_buffers():
    rng = np.random.default_rng(5)
    for t in range(1, 8):
        for X in itertools.product(range(3), repeat=t):
            X = list(X)
            S = rng.choice(np.array([0.1, 0.5, 0.5, 0.9], np.float32), size=t)
            for k in (1, 2, 3):
                o = _scan1(X, k, S, 0.3, 2, 3)
                ref = _find_all(X, k)
                assert o["count"][0] == len(ref)
                assert o["pos"][0][:len(ref)].tolist() == ref
                kept = sorted((p for p in ref if S[p] >= np.float32(0.3)),
                              key=lambda p: (-S[p], -p))[:2]
                assert o["sel_pos"][0][:len(kept)].tolist() == kept
                for c, p in enumerate(kept):
                    span = X[p + 1:p + 1 + 3]
                    assert o["sel_len"][0][c] == len(span)
                    assert o["spans"][0][c][:len(span)].tolist() == span


def test_gate_off_and_empty_key_find_nothing():
    X = [1, 2, 1, 2, 1, 2]
    o = _scan1(X, 2, np.full(6, 0.5), 0.3, 3, 2, gate_ok=np.array([0], np.uint8))
    assert o["count"][0] == 0 and o["n_sel"][0] == 0
    o = _scan1(X, 0, np.full(6, 0.5), 0.3, 3, 2)
    assert o["count"][0] == 0 and o["n_sel"][0] == 0
    o = _scan1(X, 2, np.full(6, 0.5), 0.3, 3, 2, gate_ok=np.array([1], np.uint8))
    assert o["count"][0] == 2


def test_position_capacity_truncates_but_selection_sees_all():
    X = [3] * 40
    S = np.full(40, 0.5, np.float32)
    S[2] = 0.95  # beyond the stored positions' reach it would still be chosen
    o = _scan1(X, 1, S, 0.3, 2, 2, pos_cap=5)
    assert o["count"][0] == 39
    assert o["pos"][0].tolist() == [0, 1, 2, 3, 4]
    assert o["status"][0] & oracle.ST_TRUNCATED
    assert o["sel_pos"][0].tolist() == [2, 38]
    # the same buffer with ample capacity sets no status
    o = _scan1(X, 1, S, 0.3, 2, 2, pos_cap=64)
    assert o["status"][0] == 0


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_planted_origins_are_found(name):
    w = synth.make(name)
    p = w.params()
    for b in range(w.B):
        t0, t1 = w.tok_off[b], w.tok_off[b + 1]
        X = w.tokens[t0:t1]
        for k in range(1, p["l"] + 1):
            o = _scan1(X, k, np.full(X.size, 0.5), 0.3, p["top_c"], p["span_len"], pos_cap=4096)
            ref = _find_all(X.tolist(), k)
            assert o["pos"][0][:o["count"][0]].tolist() == ref
            for origin in w.sel_pos[b]:
                if origin >= 0:
                    assert origin in ref


def test_requests_are_independent():
    # request 1's buffer repeats request 0's key but must not match across
    X0 = [1, 2, 3, 1, 2]
    X1 = [9, 1, 2, 8, 8]
    tokens = np.array(X0 + X1, np.int32)
    o = oracle.match_scan(tokens, np.array([0, 5, 10]), np.array([2, 1]), np.full(10, 0.5),
                          0.3, 2, 2, 8)
    assert o["count"].tolist() == [1, 1]
    assert o["pos"][0][:1].tolist() == [1] and o["pos"][1][:1].tolist() == [3]
