"""Pins of the sampling oracle (Section 3.4, drafter outputs: lossless
speculative sampling over the model-drafted nodes).

The draw is checked against closed forms (uniform and one-hot rows), an exact
stratified histogram (n evenly spaced uniforms give every token n p(v)
draws up to one), the temperature identity softmax(z / 0.5) = softmax(2 z),
and hand-built trees whose walks are known.
"""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore")


def test_uniform_row_inverts_exactly():
    V = 1000
    z = np.zeros(V, np.float32)
    for k in (0, 1, 17, 499, 998, 999):
        assert oracle.sample_row(z, 1.0, (k + 0.5) / V) == k
    assert oracle.sample_row(z, 1.0, 0.0) == 0


def test_one_hot_and_masked_rows():
    z = np.full(50, -np.inf, np.float32)
    z[31] = 2.0
    for u in (0.0, 0.3, 0.999999):
        assert oracle.sample_row(z, 0.7, u) == 31
    # masked tokens are never drawn: mass only on ids 3 and 40
    z = np.full(64, -np.inf, np.float32)
    z[3], z[40] = 0.0, 0.0
    assert oracle.sample_row(z, 1.0, 0.25) == 3
    assert oracle.sample_row(z, 1.0, 0.75) == 40


@pytest.mark.parametrize("T", [1.0, 0.6, 2.5])
def test_stratified_histogram_matches_the_law(T):
    # n uniforms (i + 1/2)/n hit token v exactly floor or ceil of n p(v) times
    # (up to one more at each CDF edge), whatever p is
    rng = np.random.default_rng(3)
    z = (rng.standard_normal(7) * 2).astype(np.float32)
    p = np.exp((z.astype(np.float64) - z.max()) / T)
    p /= p.sum()
    n = 7000
    counts = np.bincount([oracle.sample_row(z, T, (i + 0.5) / n) for i in range(n)], minlength=7)
    assert np.all(np.abs(counts - n * p) <= 1.0 + 1e-9), (counts, n * p)


def test_order_is_token_id_order():
    # two tokens of equal mass: the lower id takes the lower half of [0, 1)
    z = np.array([-np.inf, 1.0, -np.inf, 1.0], np.float32)
    assert oracle.sample_row(z, 1.0, 0.49) == 1
    assert oracle.sample_row(z, 1.0, 0.51) == 3


def test_temperature_is_a_logit_scale():
    rng = np.random.default_rng(5)
    z = (rng.standard_normal(300) * 3).astype(np.float32)
    for u in rng.random(50):
        assert oracle.sample_row(z, 0.5, u) == oracle.sample_row(2 * z, 1.0, u)


def _one_hot_rows(V, ids):
    L = np.full((len(ids), V), -np.inf, np.float32)
    for r, v in enumerate(ids):
        L[r, v] = 0.0
    return L


def test_walk_follows_model_children_and_stops_with_the_correction():
    # root(0) -> model 1 (tok 5), model 2 (tok 7), retrieved 3 (tok 9) ;
    # 2 -> model 4 (tok 1)
    parents = np.array([-1, 0, 0, 0, 2], np.int32)
    source = np.array([0, 1, 1, 2, 1], np.uint8)
    tokens = np.array([0, 5, 7, 9, 1], np.int32)
    node_off = np.array([0, 5], np.int32)
    u = np.full(5, 0.5)
    # root draws 7 -> node 2; node 2 draws 1 -> node 4; node 4 draws 3 (no child)
    L = _one_hot_rows(10, [7, 0, 1, 0, 3])
    o = oracle.tree_sample(L, node_off, tokens, parents, source, 1.0, u, acc_cap=4)
    assert list(o["draw"]) == [7, 0, 1, 0, 3]
    assert o["acc_len"][0] == 2 and list(o["acc_nodes"][0]) == [2, 4, -1, -1]
    assert o["bonus"][0] == 3 and o["status"][0] == 0
    # a retrieved child with the drawn token is not a model proposal: root draws 9
    L = _one_hot_rows(10, [9, 0, 1, 0, 3])
    o = oracle.tree_sample(L, node_off, tokens, parents, source, 1.0, u, acc_cap=4)
    assert o["acc_len"][0] == 0 and o["bonus"][0] == 9
    # capacity: the path is longer than acc_cap
    L = _one_hot_rows(10, [7, 0, 1, 0, 3])
    o = oracle.tree_sample(L, node_off, tokens, parents, source, 1.0, u, acc_cap=1)
    assert o["acc_len"][0] == 2 and list(o["acc_nodes"][0]) == [2]
    assert o["status"][0] == oracle.ST_TRUNCATED


def test_first_emitted_token_has_the_target_law():
    # whatever the tree, the first emitted token (first accepted child's token,
    # else the correction) is the root's draw: stratified uniforms on the root
    # give the root law up to one count per token
    rng = np.random.default_rng(8)
    V, n = 6, 6000
    parents = np.array([-1, 0, 0, 1], np.int32)
    source = np.array([0, 1, 1, 1], np.uint8)
    tokens = np.array([0, 2, 4, 5], np.int32)
    zr = (rng.standard_normal(V) * 1.5).astype(np.float32)
    L = np.tile(zr, (4, 1))
    p = np.exp((zr.astype(np.float64) - zr.max()) / 0.8)
    p /= p.sum()
    first = []
    for i in range(n):
        u = np.array([(i + 0.5) / n, 0.5, 0.5, 0.5])
        o = oracle.tree_sample(L, np.array([0, 4], np.int32), tokens, parents, source, 0.8, u, 4)
        first.append(tokens[o["acc_nodes"][0][0]] if o["acc_len"][0] > 0 else o["bonus"][0])
    counts = np.bincount(first, minlength=V)
    assert np.all(np.abs(counts - n * p) <= 1.0 + 1e-9), (counts, n * p)


def test_malformed_tree_is_rejected():
    parents = np.array([-1, 0, 5], np.int32)   # 5 >= own index
    source = np.array([0, 1, 1], np.uint8)
    o = oracle.tree_sample(_one_hot_rows(4, [1, 2, 3]), np.array([0, 3], np.int32),
                           np.array([0, 1, 2], np.int32), parents, source, 1.0, np.full(3, 0.5), 4)
    assert o["status"][0] == oracle.ST_BAD_TREE and o["acc_len"][0] == 0 and o["bonus"][0] == -1
    assert list(o["draw"]) == [1, 2, 3]
