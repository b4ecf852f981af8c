"""Pins for the oracle's entropy and trigger (Section 3.2.1, Eq. 1-3).

Each check ties the oracle to something other than itself: closed forms of
the entropy, invariances of the definition, scipy's entropy routine and
hand-worked gate cases (tests/golden/gate_cases.json).
"""
import json
import math
import os

import numpy as np
import pytest

import oracle


@pytest.mark.parametrize("V", [1024, 32000, 128256])
def test_uniform_is_log_v(V):
    # uniform distribution over V symbols: H = ln V nats, up to the fp64
    # summation bound V * 2^-53 of the oracle's plain sums
    assert oracle.row_entropy(np.full(V, 0.375, np.float32)) == pytest.approx(math.log(V), rel=V * 2.0**-52)


@pytest.mark.parametrize("V", [2, 1024, 32000])
def test_one_hot_is_zero(V):
    z = np.full(V, -np.inf, np.float32)
    z[V // 3] = 0.0
    assert oracle.row_entropy(z) == 0.0
    z = np.zeros(V, np.float32)
    z[1] = 1e4  # exp(-1e4) underflows: every other probability is exactly 0
    assert oracle.row_entropy(z) == 0.0


@pytest.mark.parametrize("V,n,a,b", [(1024, 1, 3.0, 0.0), (32000, 7, 1.0, -2.0), (128256, 100, 0.0, -5.0)])
def test_two_level_closed_form(V, n, a, b):
    # n logits at a, V-n at b: Z = n e^a + (V-n) e^b, H = ln Z - (n a e^a + (V-n) b e^b)/Z
    z = np.full(V, b, np.float32)
    z[:n] = a
    Z = n * math.exp(a) + (V - n) * math.exp(b)
    H = math.log(Z) - (n * a * math.exp(a) + (V - n) * b * math.exp(b)) / Z
    assert oracle.row_entropy(z) == pytest.approx(H, rel=V * 2.0**-52, abs=1e-12)


def test_three_symbol_closed_form():
    # logits (1, 0, 0): p = (e, 1, 1)/(e+2), H = ln(e+2) - e/(e+2)
    e = math.e
    H = math.log(e + 2) - e / (e + 2)
    assert oracle.row_entropy(np.array([1.0, 0.0, 0.0], np.float32)) == pytest.approx(H, rel=1e-14)
    # logits (ln 2, 0, 0) -> p = (1/2, 1/4, 1/4), H = 1.5 ln 2 (float32(ln 2) is off by ~1e-8)
    z = np.array([math.log(2.0), 0.0, 0.0], np.float32)
    assert oracle.row_entropy(z) == pytest.approx(1.5 * math.log(2.0), rel=1e-7)


def test_matches_scipy_on_random_rows():
    from scipy.special import softmax
    from scipy.stats import entropy
    rng = np.random.default_rng(1)
    for V, s in [(50, 0.1), (1000, 2.0), (32000, 6.0)]:
        z = (rng.standard_normal(V) * s).astype(np.float32)
        ref = entropy(softmax(z.astype(np.float64)))
        assert oracle.row_entropy(z) == pytest.approx(ref, rel=1e-11, abs=1e-12)


def test_shift_and_permutation_invariance():
    rng = np.random.default_rng(2)
    z = (rng.standard_normal(5000) * 3).astype(np.float32)
    h = oracle.row_entropy(z)
    # shifting by a power of two keeps the fp32 values' differences exact
    assert oracle.row_entropy(z + np.float32(256.0)) == pytest.approx(h, rel=1e-6)
    assert oracle.row_entropy(rng.permutation(z)) == pytest.approx(h, rel=1e-12)


def test_entropy_grows_with_temperature():
    rng = np.random.default_rng(3)
    g = rng.standard_normal(4000).astype(np.float32)
    hs = [oracle.row_entropy(g * np.float32(b)) for b in (8.0, 4.0, 2.0, 1.0, 0.5, 0.0)]
    assert all(x < y for x, y in zip(hs, hs[1:]))
    assert hs[-1] == pytest.approx(math.log(4000), rel=1e-12)


def test_rows_match_single_row():
    rng = np.random.default_rng(4)
    L = (rng.standard_normal((5, 300)) * 2).astype(np.float32)
    H = oracle.entropy_rows(L)
    for r in range(5):
        assert H[r] == oracle.row_entropy(L[r])


def _gate_case(c):
    l = c["l"]
    H = np.zeros(0)
    return oracle.gate(H, np.array([0, 0]), np.zeros(0, np.uint8), np.array([c["hist"]]),
                       np.array([c["hist_n"]]), l, c["lambda_e"], c["theta"])


def test_gate_golden(golden_dir):
    cases = json.load(open(os.path.join(golden_dir, "gate_cases.json")))
    for c in cases["cases"]:
        g = _gate_case(c)
        assert g["k_star"][0] == c["k_star"], c["name"]
        hb = math.inf if c["h_best"] == "inf" else c["h_best"]
        assert g["h_best"][0] == pytest.approx(hb, rel=1e-15), c["name"]
        assert g["ok"][0] == c["ok"], c["name"]


def test_gate_history_push(golden_dir):
    p = json.load(open(os.path.join(golden_dir, "gate_cases.json")))["push"]
    H = np.array(p["H"], np.float64)
    g = oracle.gate(H, np.array([0, len(H)]), np.array(p["row_commit"], np.uint8),
                    np.array([p["hist"]]), np.array([p["hist_n"]]), p["l"], 0.5, 1.5)
    assert g["hist"][0].tolist() == p["hist_after"]
    assert g["hist_n"][0] == p["hist_n_after"]
    # a partly filled history grows instead of shifting
    g = oracle.gate(H, np.array([0, len(H)]), np.array([0, 1, 0, 0, 0], np.uint8),
                    np.array([[0.5, 0.0, 0.0]]), np.array([1]), 3, 0.5, 1.5)
    assert g["hist"][0].tolist() == [0.5, 2.0, 0.0] and g["hist_n"][0] == 2


def test_gate_is_per_request():
    # two requests with different row ranges do not see each other's rows
    H = np.array([0.1, 0.2, 5.0, 6.0])
    g = oracle.gate(H, np.array([0, 2, 4]), np.ones(4, np.uint8), np.zeros((2, 2)),
                    np.array([0, 0]), 2, 0.0, 1.5)
    assert g["hist"].tolist() == [[0.1, 0.2], [5.0, 6.0]]
    # request 0: H1=0.2, H2=0.15 -> k*=2; request 1: H1=6, H2=5.5 -> k*=2
    assert g["k_star"].tolist() == [2, 2]
    assert g["ok"].tolist() == [1, 0]
