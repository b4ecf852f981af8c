"""GPU parity of rs_tree_sample (Section 3.4, drafter outputs: lossless
speculative sampling) against the oracle.

Draws: the GPU evaluates the inverse CDF in fp32 (per-thread sums of 32
consecutive ids, a block scan, chunk weights rescaled to the row maximum),
the oracle in fp64 in plain id order.  A uniform that falls within the
accumulated rounding of a CDF step may land on the neighbouring token, so
every draw must either equal the oracle's or be a valid draw of the fp64 law
within CDF_EPS, and mismatches must stay rare.  CDF_EPS bounds the relative
error of an fp32 partial sum here: ex2.approx (2 ulp) on each term, 32-term
sequential thread sums (32 ulp), a 13-step block scan and the chunk
rescaling, about 50 ulp of 2^-24 in all, i.e. 3e-6 of the row mass; 2e-5
leaves margin for the fp32 temperature scale.
Walk: the oracle is re-run on the GPU's own draws (one-hot rows that carry
them), so the accepted path, its length, the correction token and the status
are compared exactly.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2511_01282_gb300 import respec as rs

pytestmark = pytest.mark.gpu

CDF_EPS = 2e-5
MISMATCH_FRAC = 0.01


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_gpu(logits, node_off, tokens, parents, source, T, u, acc_cap):
    R, V = logits.shape
    B = len(node_off) - 1
    i32 = lambda *s: torch.full(s, -7, dtype=torch.int32, device="cuda")  # noqa: E731
    out = dict(draw=i32(max(R, 1)), acc_len=i32(B), acc_nodes=i32(B, acc_cap), bonus=i32(B), status=i32(B))
    ws = torch.empty(max(rs.rs_tree_sample_workspace_size(R, V), 256), dtype=torch.uint8, device="cuda")
    rs.rs_tree_sample(_cuda(logits), R, V, _cuda(node_off), B, _cuda(tokens), _cuda(parents), _cuda(source),
                      T, _cuda(u.astype(np.float32)), acc_cap, out["draw"], out["acc_len"], out["acc_nodes"],
                      out["bonus"], out["status"], ws)
    torch.cuda.synchronize()
    o = {k: v.cpu().numpy() for k, v in out.items()}
    o["draw"] = o["draw"][:R]
    return o


def valid_draw(z, T, u, v):
    z = z.astype(np.float64)
    m = z.max()
    if m == -np.inf:
        return v == 0
    p = np.exp((z - m) / T)
    cdf = np.cumsum(p) / p.sum()
    lo = cdf[v - 1] if v > 0 else 0.0
    if u >= 1.0:  # the last id with mass
        return v == np.nonzero(p > 0)[0][-1]
    return p[v] > 0 and lo <= u + CDF_EPS and cdf[v] >= u - CDF_EPS


def check(logits, node_off, tokens, parents, source, T, u, acc_cap=32):
    u = np.asarray(u, np.float32)
    got = run_gpu(logits, node_off, tokens, parents, source, np.float32(T), u, acc_cap)
    ref = oracle.tree_sample(logits, node_off, tokens, parents, source, float(np.float32(T)),
                             u.astype(np.float64), acc_cap)
    bad = np.nonzero(got["draw"] != ref["draw"])[0]
    assert len(bad) <= max(2, MISMATCH_FRAC * len(u)), "%d of %d draws differ" % (len(bad), len(u))
    for r in bad:
        assert valid_draw(logits[r], float(np.float32(T)), float(u[r]), int(got["draw"][r])), \
            "row %d: draw %d vs %d is not a valid draw" % (r, got["draw"][r], ref["draw"][r])
    # the walk, on the GPU's own draws: one-hot rows over a compact id space
    # (only equality between a draw and a child's token matters)
    ids, inv = np.unique(np.concatenate([got["draw"], np.asarray(tokens)]), return_inverse=True)
    d_c, t_c = inv[:len(u)], inv[len(u):].astype(np.int32)
    onehot = np.full((len(u), len(ids)), -np.inf, np.float32)
    onehot[np.arange(len(u)), d_c] = 0.0
    walk = oracle.tree_sample(onehot, node_off, t_c, parents, source, 1.0, np.full(len(u), 0.5), acc_cap)
    walk["bonus"] = np.where(walk["bonus"] >= 0, ids[np.maximum(walk["bonus"], 0)], -1)
    for k in ("acc_len", "acc_nodes", "bonus", "status"):
        assert (got[k] == walk[k]).all(), k
    return got, ref


def _uniforms(rng, R):
    u = rng.random(R).astype(np.float32)
    if R >= 4:
        u[0] = 0.0
        u[1] = np.nextafter(np.float32(1.0), np.float32(0.0))
        u[2] = 1.0          # >= 1: the last id with mass
    return u


@pytest.mark.parametrize("name,T", [("tiny", 1.0), ("7b", 0.7), ("7b", 2.0)])
def test_named_workloads(name, T):
    w = synth.make(name)
    rng = np.random.default_rng(11)
    got, _ = check(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, T, _uniforms(rng, w.R))
    assert (got["status"] == 0).all()


@pytest.mark.parametrize("V", [1001, 4096, 8192, 8193, 50000])
def test_vocab_sizes_and_alignment(V):
    # V % 4 != 0 takes the scalar path; 8192 / 8193 straddle the chunk size
    w = synth.build(synth.small_spec(B=3, V=V), seed=V)
    rng = np.random.default_rng(V)
    check(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, 1.0, _uniforms(rng, w.R))


def test_masked_and_empty_rows():
    w = synth.build(synth.small_spec(B=2, V=3000), seed=4)
    L = w.logits.copy()
    L[1, :2500] = -np.inf            # mass only on the tail
    L[2, :] = -np.inf                # no mass: draw 0
    L[3, :] = -np.inf
    L[3, 1234] = 5.0                 # one-hot
    rng = np.random.default_rng(4)
    got, _ = check(L, w.node_off, w.tree_tokens, w.parents, w.source, 0.5, _uniforms(rng, w.R))
    assert got["draw"][2] == 0 and got["draw"][3] == 1234


def test_walk_accepts_planted_children_and_truncates():
    # request 0: root -> 1 -> 2 -> 3 -> 4, all model nodes; request 1: root ->
    # model 1 (tok 11), model 2 (tok 12), retrieved 3 -> 4.  Each row puts
    # nearly all its mass on one token, so the walks are known.
    V = 700
    parents = np.array([-1, 0, 1, 2, 3, -1, 0, 0, 0, 3], np.int32)
    source = np.array([0, 1, 1, 1, 1, 0, 1, 1, 2, 2], np.uint8)
    tokens = np.array([5, 21, 22, 23, 24, 6, 11, 12, 13, 14], np.int32)
    node_off = np.array([0, 5, 10], np.int32)
    L = np.full((10, V), -3.0, np.float32)
    for r, t in enumerate([21, 22, 23, 24, 99, 12, 300, 301, 302, 303]):
        L[r, t] = 30.0
    rng = np.random.default_rng(6)
    got, _ = check(L, node_off, tokens, parents, source, 1.0, rng.random(10), acc_cap=2)
    assert list(got["acc_len"]) == [4, 1] and list(got["bonus"]) == [99, 301]
    assert list(got["acc_nodes"][0]) == [1, 2] and list(got["acc_nodes"][1]) == [2, -1]
    assert got["status"][0] == rs.RS_ST_TRUNCATED and got["status"][1] == 0


def test_bad_tree_status():
    w = synth.build(synth.small_spec(B=2, V=500), seed=7)
    par = w.parents.copy()
    par[w.node_off[1] + 2] = 99   # request 1: a parent after the node
    rng = np.random.default_rng(7)
    got, _ = check(w.logits, w.node_off, w.tree_tokens, par, w.source, 1.0, rng.random(w.R))
    assert got["status"][1] == rs.RS_ST_BAD_TREE and got["acc_len"][1] == 0 and got["bonus"][1] == -1
    assert got["status"][0] == 0


@pytest.mark.slow
@pytest.mark.parametrize("name", ["13b32k", "batched"])
def test_full_size(name):
    w = synth.make(name)
    rng = np.random.default_rng(13)
    check(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, 1.0, _uniforms(rng, w.R))
