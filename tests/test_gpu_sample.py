"""GPU parity of rs_tree_sample (Section 3.4, drafter outputs: lossless
speculative sampling) against the oracle.

Draws: every draw must equal the oracle's fp64 inverse CDF.  The GPU settles
most rows in fp32 under a rigorous error bound and redoes the rest in fp64,
so the only freedom left is rounding at the 1e-13 level: a draw may differ
only where u Z lies within (V 2^-52 + 2^-40) Z of a CDF step between the two
draws (V 2^-52: the bound on the oracle's sequential fp64 sum of V terms;
2^-40: the GPU's exact pass, double-float terms good to ~1e-14 per nat of
|z - max z| / T, summed in fp64).  The step-
straddling test puts uniforms a few fp32 ulps from CDF steps, on both sides
of the certificate's margin, so that both the fp32 certificate and the fp64
pass decide draws there; RS_DEBUG_SAMPLE_EXACT=1 sends every row through the
fp64 pass.
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


def near_step(z, T, u, a, b):
    """True when u Z lies within the oracle's fp64 rounding of every CDF step
    between draws a and b (p in fp64, summed in id order as the oracle does)."""
    z = z.astype(np.float64)
    p = np.exp((z - z.max()) / T)
    c = np.cumsum(p)
    lo, hi = min(a, b), max(a, b)
    tol = (len(z) * 2.0 ** -52 + 2.0 ** -40) * c[-1]
    return bool(np.all(np.abs(c[lo:hi] - u * c[-1]) <= tol))


def check(logits, node_off, tokens, parents, source, T, u, acc_cap=32):
    u = np.asarray(u, np.float32)
    got = run_gpu(logits, node_off, tokens, parents, source, np.float32(T), u, acc_cap)
    ref = oracle.tree_sample(logits, node_off, tokens, parents, source, float(np.float32(T)),
                             u.astype(np.float64), acc_cap)
    bad = np.nonzero(got["draw"] != ref["draw"])[0]
    for r in bad:
        assert near_step(logits[r], float(np.float32(T)), float(u[r]), int(got["draw"][r]), int(ref["draw"][r])), \
            "row %d: draw %d, oracle %d (u = %r)" % (r, got["draw"][r], ref["draw"][r], float(u[r]))
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


@pytest.mark.parametrize("V", [1001, 4096, 8192, 8193, 50000, 270000])
def test_vocab_sizes_and_alignment(V):
    # V % 4 != 0 takes the scalar path; 8192 / 8193 straddle the chunk size;
    # 270000 has more than 32 chunks (the two-round chunk scan)
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


def _step_uniforms(z, T, steps, ulps=(-64, -16, -4, -1, 0, 1, 4, 16, 64)):
    """fp32 uniforms a few ulps either side of the CDF steps after the given
    ids (fp64 CDF in id order)."""
    z = z.astype(np.float64)
    p = np.exp((z - z.max()) / T)
    c = np.cumsum(p) / p.sum()
    out = []
    for k in steps:
        u0 = np.float32(c[k])
        for d in ulps:
            u = u0
            for _ in range(abs(d)):
                u = np.nextafter(u, np.float32(np.inf if d > 0 else -np.inf))
            if 0.0 <= u < 1.0:
                out.append(u)
    return np.array(out, np.float32)


@pytest.mark.parametrize("kind", ["flat", "gauss", "peaked"])
def test_uniforms_at_cdf_steps(kind):
    # rows whose CDF steps are dense (flat: 1/V apart) or uneven; each row is
    # repeated once per uniform, the uniforms a few fp32 ulps from a step
    V = 20000
    rng = np.random.default_rng(17)
    z = {"flat": np.zeros(V, np.float32),
         "gauss": rng.standard_normal(V).astype(np.float32) * 2,
         "peaked": rng.standard_normal(V).astype(np.float32) * 8}[kind]
    T = 1.0
    steps = rng.choice(V - 1, 24, replace=False)
    u = _step_uniforms(z, T, steps)
    R = len(u)
    L = np.tile(z, (R, 1))
    node_off = np.arange(R + 1, dtype=np.int32)          # one root-only request per row
    tokens = np.zeros(R, np.int32)
    parents = np.full(R, -1, np.int32)
    source = np.zeros(R, np.uint8)
    got, ref = check(L, node_off, tokens, parents, source, T, u)
    assert (got["draw"] == ref["draw"]).all()


def test_fp64_tail_below_fp32_range():
    # the only mass after id 3000 sits 100 nats below the maximum: 2^-144 in
    # fp32 units (flushed) but exp(-100) in fp64, so the last id with mass
    # (u >= 1) and draws next to it come from the fp64 pass
    V = 4000
    z = np.full(V, -np.inf, np.float32)
    z[:3000] = np.random.default_rng(3).standard_normal(3000).astype(np.float32)
    z[3001] = z[:3000].max() - 100.0
    z[3500] = z[:3000].max() - 101.0
    u = np.array([0.0, 0.25, 0.5, np.nextafter(np.float32(1), np.float32(0)), 1.0], np.float32)
    R = len(u)
    L = np.tile(z, (R, 1))
    node_off = np.arange(R + 1, dtype=np.int32)
    got, ref = check(L, node_off, np.zeros(R, np.int32), np.full(R, -1, np.int32), np.zeros(R, np.uint8), 1.0, u)
    assert (got["draw"] == ref["draw"]).all()
    assert got["draw"][-1] == 3500


def test_tiny_uniforms_reach_terms_below_fp32_range():
    # u = 0 and fp32 uniforms down to the smallest subnormal: u Z falls among
    # leading terms 90-120 nats below the maximum, which only fp64 represents
    V = 3000
    z = np.random.default_rng(5).standard_normal(V).astype(np.float32)
    M = z.max()
    z[0], z[1], z[2] = M - 120.0, M - 100.0, M - 90.0
    tiny = np.float32(np.finfo(np.float32).smallest_subnormal)
    u = np.array([0.0, tiny, tiny * 64, 1e-41, 1e-38, 2.0 ** -41, 2.0 ** -30, 0.5], np.float32)
    R = len(u)
    L = np.tile(z, (R, 1))
    node_off = np.arange(R + 1, dtype=np.int32)
    got, ref = check(L, node_off, np.zeros(R, np.int32), np.full(R, -1, np.int32), np.zeros(R, np.uint8), 1.0, u)
    assert (got["draw"] == ref["draw"]).all()
    assert got["draw"][0] == 0 and len(set(ref["draw"][:5])) >= 3  # the walk stopped at different leading ids


@pytest.mark.parametrize("name,T", [("tiny", 1.0), ("7b", 0.7), ("7b", 2.0)])
def test_every_row_through_the_fp64_pass(name, T, monkeypatch):
    monkeypatch.setenv("RS_DEBUG_SAMPLE_EXACT", "1")
    w = synth.make(name)
    rng = np.random.default_rng(23)
    got, ref = check(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, T, _uniforms(rng, w.R))
    assert (got["draw"] == ref["draw"]).all()


@pytest.mark.parametrize("V", [1, 255, 257, 8193])
def test_fp64_pass_slice_edges(V, monkeypatch):
    monkeypatch.setenv("RS_DEBUG_SAMPLE_EXACT", "1")
    w = synth.build(synth.small_spec(B=2, V=max(V, 300)), seed=V)
    L = w.logits[:, :V].copy()
    rng = np.random.default_rng(V)
    check(L, w.node_off, np.minimum(w.tree_tokens, V - 1), w.parents, w.source, 1.0, _uniforms(rng, w.R))
