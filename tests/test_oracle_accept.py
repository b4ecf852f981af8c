"""Pins for the oracle's verification, path selection and EMA update.

Section 3.4 (Eq. 6-7, look-ahead tolerance), Eq. 4-5 and Algorithm 1's
verification and score update.  Checked against hand-worked look-ahead cases
(tests/golden/lookahead_cases.json), numpy's lexicographic sort and scipy's
log-softmax for the row statistics, brute-force path enumeration for the
model tree, the reductions the definition implies (phi = 0 or beta = 1 is
strict verification) and the closed form of repeated EMA updates.
"""
import json
import os

import numpy as np
import pytest
from scipy.special import log_softmax, logsumexp

import oracle
import synth


def _rows(case_rows, V):
    z = np.zeros((len(case_rows), V), np.float32)
    for r, d in enumerate(case_rows):
        for k, val in d.items():
            z[r, int(k)] = val
    return z


def _chain_request(tokens, rows, sel=5, t=20):
    """Single request: root + one retrieved chain (chain id 0)."""
    L = len(tokens)
    return dict(logits=rows, node_off=np.array([0, L + 1]), tokens=np.array([0] + tokens),
                parents=np.array([-1] + list(range(L))), source=np.array([0] + [2] * L),
                chain=np.array([-1] + [0] * L), sel_pos=np.array([[sel, -1, -1]]),
                tok_off=np.array([0, t]), scores=np.full(t, 0.5, np.float32))


def _accept(req, beta, tau, phi, m, alpha=0.3, acc_cap=16):
    return oracle.accept(req["logits"], req["node_off"], req["tokens"], req["parents"],
                         req["source"], req["chain"], req["sel_pos"], req["tok_off"],
                         req["scores"], beta, tau, phi, m, alpha, acc_cap)


def test_lookahead_golden(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "lookahead_cases.json")))
    for c in g["cases"]:
        req = _chain_request(c["tokens"], _rows(c["rows"], g["V"]))
        o = _accept(req, g["beta"], g["tau"], c["phi"], c["m"])
        L = len(c["tokens"])
        assert o["acc_len"][0] == c["acc_len"], c["name"]
        assert o["bonus"][0] == c["bonus"], c["name"]
        assert o["winner"][0] == (0 if c["acc_len"] > 0 else -2), c["name"]
        assert o["acc_nodes"][0][:c["acc_len"]].tolist() == list(range(1, c["acc_len"] + 1))
        assert o["commit"].tolist() == [1] + [1 if j < c["acc_len"] else 0 for j in range(L)]
        # Eq. 4-5: winner gets R = L_acc / L_draft, otherwise R = 0
        R = c["acc_len"] / L
        assert o["scores"][5] == np.float32(0.7 * 0.5 + 0.3 * R), c["name"]
        assert o["status"][0] == 0


def test_row_statistics_against_library_routines():
    rng = np.random.default_rng(11)
    V, R, beta = 257, 40, 7
    z = np.round(rng.standard_normal((R, V)) * 4, 1).astype(np.float32)  # many exact ties
    req = dict(logits=z, node_off=np.array([0, R]), tokens=np.zeros(R, np.int32),
               parents=np.arange(-1, R - 1), source=np.array([0] + [1] * (R - 1)),
               chain=np.full(R, -1), sel_pos=np.full((1, 3), -1), tok_off=np.array([0, 4]),
               scores=np.zeros(4, np.float32))
    req["tokens"] = rng.integers(0, V, R)
    o = _accept(req, beta, 1.0, 2, 2)
    for r in range(R):
        order = np.lexsort((np.arange(V), -z[r].astype(np.float64)))  # logit desc, id asc
        assert o["topk"][r].tolist() == order[:beta].tolist()
        assert o["argmax"][r] == order[0]
        assert o["lse"][r] == pytest.approx(logsumexp(z[r].astype(np.float64)), rel=1e-14)
    for i in range(1, R):
        ref = np.exp(log_softmax(z[i - 1].astype(np.float64))[req["tokens"][i]])
        assert o["p_tok"][i] == pytest.approx(ref, rel=1e-12)
    assert o["p_tok"][0] == 1.0


def test_relaxed_check_is_eq7_on_log_probabilities():
    # a one-token chain with phi = 1, m = 0 is accepted iff the token passes
    # Eq. 6 and Eq. 7 (or is greedy); compare with scipy's log-softmax
    rng = np.random.default_rng(12)
    V, beta = 64, 4
    for trial in range(300):
        tau = float(np.float32(rng.uniform(0, 3)))
        z = (rng.standard_normal((2, V)) * rng.uniform(0.5, 4)).astype(np.float32)
        tok = int(rng.integers(0, V))
        if trial % 3 == 0:
            order = np.lexsort((np.arange(V), -z[0].astype(np.float64)))
            tok = int(order[rng.integers(0, 6)])
        req = _chain_request([tok], z)
        o = _accept(req, beta, tau, 1, 0)
        lp = log_softmax(z[0].astype(np.float64))
        order = np.lexsort((np.arange(V), -z[0].astype(np.float64)))
        gap = lp[order[0]] - lp[tok]
        if abs(gap - tau) < 1e-9:
            continue
        expect = tok in order[:beta].tolist() and gap <= tau
        assert o["acc_len"][0] == int(expect)


def test_phi_zero_and_beta_one_are_strict():
    for name in ("tiny", "7b"):
        w = synth.make(name)
        p = w.params()
        base = dict(logits=w.logits, node_off=w.node_off, tokens=w.tree_tokens, parents=w.parents,
                    source=w.source, chain=w.chain, sel_pos=w.sel_pos, tok_off=w.tok_off,
                    scores=w.scores)
        strict = _accept(base, 1, 0.0, 0, 0)
        for beta, tau, phi, m in [(p["beta"], p["tau"], 0, p["m"]), (1, p["tau"], 3, 0)]:
            o = _accept(base, beta, tau, phi, m)
            assert o["acc_len"].tolist() == strict["acc_len"].tolist()
            assert o["winner"].tolist() == strict["winner"].tolist()
        # strict chain length is the greedy prefix: brute force
        N = int(w.node_off[1])
        am = strict["argmax"]
        for c in range(p["top_c"]):
            nodes = [i for i in range(N) if w.chain[i] == c]
            l0 = 0
            while l0 < len(nodes) and w.tree_tokens[nodes[l0]] == am[w.parents[nodes[l0]]]:
                l0 += 1
            if strict["winner"][0] == c:
                assert strict["acc_len"][0] == l0
            else:
                assert l0 <= strict["acc_len"][0]


def _brute_model_path(parents, tokens, source, argmax):
    """Longest all-greedy model path by enumerating every root-to-node path."""
    N = len(parents)
    best, best_node = 0, 0
    for i in range(1, N):
        if source[i] != 1:
            continue
        path = []
        a = i
        while a > 0:
            path.append(a)
            a = parents[a]
        if all(tokens[x] == argmax[parents[x]] for x in path) and len(path) > best:
            best, best_node = len(path), i
    return best, best_node


@pytest.mark.parametrize("seed", range(6))
def test_model_tree_longest_path_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    V, N = 6, 40
    parents = np.array([-1] + [int(rng.integers(0, i)) for i in range(1, N)])
    z = rng.integers(0, 4, (N, V)).astype(np.float32)  # small alphabet: many greedy hits and ties
    tokens = rng.integers(0, V, N)
    req = dict(logits=z, node_off=np.array([0, N]), tokens=tokens, parents=parents,
               source=np.array([0] + [1] * (N - 1)), chain=np.full(N, -1),
               sel_pos=np.full((1, 3), -1), tok_off=np.array([0, 4]), scores=np.zeros(4, np.float32))
    o = _accept(req, 3, 1.0, 2, 1, acc_cap=N)
    best, node = _brute_model_path(parents, tokens, req["source"], o["argmax"])
    assert o["acc_len"][0] == best
    assert o["winner"][0] == (-1 if best else -2)
    if best:
        path = []
        a = node
        while a > 0:
            path.append(a)
            a = parents[a]
        assert o["acc_nodes"][0][:best].tolist() == path[::-1]
        assert o["bonus"][0] == o["argmax"][node]
        assert sorted(np.nonzero(o["commit"])[0].tolist()) == sorted([0] + path)


def test_winner_ties_and_ema_of_losers():
    # root row: id 1 greedy (model node 1), id 2 close (chain 0 head) ;
    # model node 2 greedy under node 1 -> model length 2;
    # chain 0: relaxed head + 1 greedy follower with m = 1 -> length 2 (tie -> model);
    # chain 1: one greedy token -> length 1
    V = 8
    z = np.zeros((7, V), np.float32)
    z[0, 1], z[0, 2] = 5.0, 4.5     # root row
    z[1, 3] = 5.0                   # row of model node 1
    z[2, 0] = 5.0                   # row of model node 2 (bonus 0)
    z[3, 4] = 5.0                   # row of chain-0 node 3
    z[4, 6] = 5.0
    z[5, 0] = 5.0                   # row of chain-1 node 5
    tokens = [9, 1, 3, 2, 4, 1, 0]
    tokens[0] = 0
    parents = [-1, 0, 1, 0, 3, 0, 5]
    source = [0, 1, 1, 2, 2, 2, 2]
    chain = [-1, -1, -1, 0, 0, 1, 1]
    tokens[6] = 7                   # chain 1 second token misses (row 5 argmax 0)
    req = dict(logits=z, node_off=np.array([0, 7]), tokens=np.array(tokens), parents=np.array(parents),
               source=np.array(source), chain=np.array(chain), sel_pos=np.array([[3, 8, -1]]),
               tok_off=np.array([0, 12]), scores=np.full(12, 0.5, np.float32))
    o = _accept(req, 3, 1.0, 1, 1)
    assert o["acc_len"][0] == 2 and o["winner"][0] == -1
    assert o["acc_nodes"][0][:2].tolist() == [1, 2]
    assert o["bonus"][0] == 0
    # neither chain won: both decay with R = 0
    assert o["scores"][3] == np.float32(0.35) and o["scores"][8] == np.float32(0.35)
    assert o["scores"][0] == np.float32(0.5)
    # make the model miss at depth 2: chain 0 (length 2) now beats it
    z2 = z.copy()
    z2[1, 3], z2[1, 5] = 0.0, 5.0
    req2 = dict(req, logits=z2)
    o = _accept(req2, 3, 1.0, 1, 1)
    assert o["winner"][0] == 0 and o["acc_len"][0] == 2
    assert o["scores"][3] == np.float32(0.7 * 0.5 + 0.3 * 1.0)
    assert o["scores"][8] == np.float32(0.35)
    # chains of equal length: the first selected wins
    z3 = z2.copy()
    z3[0, 2] = 5.0 - 0.25           # chain 0 head still only close
    tokens3 = list(tokens)
    tokens3[6] = 0                  # chain 1 becomes fully greedy: length 2
    req3 = dict(req2, logits=z3, tokens=np.array(tokens3))
    o = _accept(req3, 3, 1.0, 1, 1)
    assert o["winner"][0] == 0 and o["acc_len"][0] == 2


def test_ema_closed_form():
    # n consecutive losses: S0 (1-alpha)^n ; n consecutive full accepts:
    # 1 - (1 - S0)(1 - alpha)^n  (fp32 storage after each update)
    V = 8
    lose = _chain_request([1, 2], _rows([{"5": 5.0}, {"2": 5.0}, {"3": 5.0}], V))
    win = _chain_request([1, 2], _rows([{"1": 5.0}, {"2": 5.0}, {"3": 5.0}], V))
    for req, target in ((lose, lambda n: 0.5 * 0.7 ** n), (win, lambda n: 1 - 0.5 * 0.7 ** n)):
        s = req["scores"]
        for n in range(1, 30):
            o = _accept(dict(req, scores=s), 3, 0.0, 0, 0)
            s = o["scores"]
            assert s[5] == pytest.approx(target(n), abs=4e-7 * n)


def test_malformed_trees_are_flagged():
    V = 4
    z = np.zeros((3, V), np.float32)
    good = dict(logits=z, node_off=np.array([0, 3]), tokens=np.array([0, 1, 2]),
                parents=np.array([-1, 0, 1]), source=np.array([0, 1, 1]), chain=np.full(3, -1),
                sel_pos=np.full((1, 3), -1), tok_off=np.array([0, 4]), scores=np.zeros(4, np.float32))
    assert _accept(good, 2, 1.0, 1, 1)["status"][0] == 0
    bads = [dict(parents=np.array([-1, 2, 1])),                       # not topological
            dict(parents=np.array([0, 0, 1])),                        # root with a parent
            dict(source=np.array([0, 2, 1]), chain=np.array([-1, 0, -1])),  # model under chain
            dict(source=np.array([0, 2, 2]), chain=np.array([-1, 0, 5])),   # chain id >= top_c
            dict(source=np.array([0, 1, 3])),                         # unknown source
            dict(source=np.array([0, 2, 2]), chain=np.array([-1, 0, 1]),
                 parents=np.array([-1, 0, 1]))]                       # chain 1 not hanging from root
    for kw in bads:
        o = _accept(dict(good, **kw), 2, 1.0, 1, 1)
        assert o["status"][0] & oracle.ST_BAD_TREE, kw
        assert o["acc_len"][0] == 0 and o["winner"][0] == -2 and o["bonus"][0] == -1
        assert o["commit"].tolist() == [0, 0, 0]
    # selected position outside the buffer
    req = _chain_request([1], _rows([{"1": 5.0}, {"2": 5.0}], 4), sel=50)
    o = _accept(req, 2, 1.0, 1, 1)
    assert o["status"][0] & oracle.ST_BAD_POS


def test_acc_capacity_truncates():
    V = 4
    L = 6
    rows = _rows([{"1": 5.0}] * (L + 1), V)
    req = _chain_request([1] * L, rows)
    o = _accept(req, 2, 1.0, 1, 1, acc_cap=4)
    assert o["acc_len"][0] == L
    assert o["acc_nodes"][0].tolist() == [1, 2, 3, 4]
    assert o["status"][0] & oracle.ST_TRUNCATED
