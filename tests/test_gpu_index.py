"""GPU parity of the indexed retrieval (rs_match_index_build +
rs_match_scan_indexed) with the oracle of Section 3.3: the same outputs as
rs_match_scan, bit for bit, from an inverted index instead of a scan."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_helpers import f32
from paper_2511_01282_gb300 import respec as rs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def build_index(tokens, tok_off, V):
    B = len(tok_off) - 1
    t_total = int(tok_off[-1])
    idx = torch.empty(rs.rs_match_index_bytes(B, V, t_total), dtype=torch.uint8, device="cuda")
    rs.rs_match_index_build(_cuda(tokens), _cuda(tok_off), B, V, t_total, idx)
    return idx, t_total


def query(tokens, tok_off, ks, ok, scores, theta, top_c, span_len, pos_cap, V, t_total, idx):
    B = len(tok_off) - 1
    z = lambda *shape: torch.full(shape, -7, dtype=torch.int32, device="cuda")  # noqa: E731
    out = dict(count=z(B), pos=z(B, pos_cap), sel_pos=z(B, top_c), sel_len=z(B, top_c),
               spans=z(B, top_c, span_len), n_sel=z(B), status=z(B))
    p = rs.params(theta_score=theta, top_c=top_c, span_len=span_len)
    rs.rs_match_scan_indexed(_cuda(tokens), _cuda(tok_off), B, _cuda(ks), _cuda(ok) if ok is not None else None,
                             _cuda(scores), p, pos_cap, out["count"], out["pos"], out["sel_pos"], out["sel_len"],
                             out["spans"], out["n_sel"], out["status"], V, t_total, idx)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def compare(tokens, tok_off, ks, ok, scores, theta, top_c, span_len, pos_cap, V, idx=None, t_total=None):
    if idx is None:
        idx, t_total = build_index(tokens, tok_off, V)
    got = query(tokens, tok_off, ks, ok, scores, theta, top_c, span_len, pos_cap, V, t_total, idx)
    ref = oracle.match_scan(tokens, tok_off, ks, scores, f32(theta), top_c, span_len, pos_cap,
                            gate_ok=ok)
    for key in ("count", "pos", "sel_pos", "sel_len", "spans", "n_sel", "status"):
        assert (got[key] == ref[key]).all(), key
    return got


@pytest.mark.parametrize("name", ["tiny", "7b", "batched", "13b32k", "gqa16k"])
@pytest.mark.parametrize("k", [1, 2, 3])
def test_named_workloads(name, k):
    w = synth.make(name)
    s = w.spec
    ks = np.full(w.B, k, np.int32)
    ok = np.ones(w.B, np.uint8)
    ok[::3] = 0                                     # some requests not triggered
    compare(w.tokens, w.tok_off, ks, ok, w.scores, s.theta_score, s.top_c, s.chain_len, 64, s.V)


@pytest.mark.parametrize("dense", [False, True])
def test_long_buffers(dense):
    rng = np.random.default_rng(31 + dense)
    lens = [8192, 8193, 65537, 150001]
    V = 3 if dense else 200
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tokens = rng.integers(0, V, int(tok_off[-1])).astype(np.int32)
    for b, t in enumerate(lens):
        a = int(tok_off[b])
        for q in rng.integers(8, t - 8, 6):
            tokens[a + q - 3:a + q + 1] = tokens[a + t - 4:a + t]
    scores = rng.random(int(tok_off[-1])).astype(np.float32)
    scores[rng.random(scores.size) < 0.1] = 0.75
    got = compare(tokens, tok_off, np.array([1, 2, 3, 4], np.int32), None, scores, 0.3, 8, 16, 5000, V)
    assert (got["n_sel"] > 0).all()


def test_tail_after_the_build_and_foreign_ids():
    # index built on each request's first part, queried on the grown buffers;
    # ids outside [0, V) (negative and >= V) share a bucket and still match
    rng = np.random.default_rng(5)
    full = [rng.integers(-5, 120, n).astype(np.int32) for n in (3000, 5000, 700)]
    cut = [2000, 5000, 1]                           # request 1 untouched, request 2 almost all tail
    for f in full:                                  # plant repeats of the last 3 tokens
        for q in rng.integers(5, len(f) - 5, 4):
            f[q - 2:q + 1] = f[-3:]
    V = 100
    b_off = np.concatenate([[0], np.cumsum(cut)]).astype(np.int64)
    b_tok = np.concatenate([f[:c] for f, c in zip(full, cut)])
    idx, t_total = build_index(b_tok, b_off, V)
    tok_off = np.concatenate([[0], np.cumsum([len(f) for f in full])]).astype(np.int64)
    tokens = np.concatenate(full)
    scores = rng.random(len(tokens)).astype(np.float32)
    for k in (1, 2, 3):
        got = compare(tokens, tok_off, np.full(3, k, np.int32), None, scores, 0.2, 3, 8, 256, V,
                      idx=idx, t_total=t_total)
        assert (got["count"] > 0).all()


def test_skips_and_truncation():
    w = synth.build(synth.small_spec(B=4, repeat_prob=0.9, seg_len=(2, 4), V=50), seed=13)
    ks = np.array([1, 2, 9, 3], np.int32)             # 9 > RS_MAX_L: skipped with a status
    ok = np.array([1, 1, 1, 0], np.uint8)
    idx, t_total = build_index(w.tokens, w.tok_off, 50)
    got = query(w.tokens, w.tok_off, ks, ok, w.scores, w.spec.theta_score, w.spec.top_c, w.spec.chain_len, 3, 50,
                t_total, idx)
    ks_o = ks.copy()
    ks_o[2] = 0
    ref = oracle.match_scan(w.tokens, w.tok_off, ks_o, w.scores, f32(w.spec.theta_score), w.spec.top_c,
                            w.spec.chain_len, 3, gate_ok=ok)
    assert got["status"][2] == rs.RS_ST_TOO_LARGE
    for key in ("count", "pos", "sel_pos", "sel_len", "spans", "n_sel"):
        assert (got[key] == ref[key]).all(), key
    assert got["status"][0] & rs.RS_ST_TRUNCATED


def _grow(rng, buf, n, V, copy_prob):
    """Append n tokens to buf: copies of earlier spans (so keys recur) or fresh ids."""
    out = list(buf)
    while len(out) < len(buf) + n:
        if len(out) > 8 and rng.random() < copy_prob:
            a = int(rng.integers(0, len(out) - 4))
            out += out[a:a + int(rng.integers(2, 6))]
        else:
            out.append(int(rng.integers(0, V)))
    return np.array(out[:len(buf) + n], np.int32)


def _layout(bufs):
    tok_off = np.concatenate([[0], np.cumsum([len(x) for x in bufs])]).astype(np.int64)
    return np.concatenate(bufs).astype(np.int32), tok_off


def test_append_matches_the_oracle_after_every_step():
    # Algorithm 1's update: each step appends a few committed tokens to every
    # request's buffer and rs_match_index_append adds them to the index; after
    # every step the indexed retrieval equals the oracle's scan bit for bit
    rng = np.random.default_rng(41)
    V = 500
    bufs = [_grow(rng, np.zeros(0, np.int32), n, V, 0.5) for n in (2000, 50, 5000, 1)]
    tokens, tok_off = _layout(bufs)
    idx, t_total = build_index(tokens, tok_off, V)
    status = torch.full((4,), -1, dtype=torch.int32, device="cuda")
    for step in range(40):
        bufs = [_grow(rng, b, int(rng.integers(0, 13)), V, 0.6) for b in bufs]
        tokens, tok_off = _layout(bufs)
        rs.rs_match_index_append(_cuda(tokens), _cuda(tok_off), 4, V, t_total, idx, status)
        torch.cuda.synchronize()
        assert (status.cpu().numpy() == 0).all()
        scores = rng.random(len(tokens)).astype(np.float32)
        ks = rng.integers(1, 4, 4).astype(np.int32)
        got = compare(tokens, tok_off, ks, None, scores, 0.25, 3, 8, 64, V, idx=idx, t_total=t_total)
    assert (got["count"] > 0).any()


def test_append_overflow_then_linear_tail():
    # one id appended far beyond its room: the overflow list takes 4096
    # positions, then indexing stops (RS_ST_TRUNCATED) and the later positions
    # are tested one by one; the answers stay exact throughout and after a
    # rebuild
    rng = np.random.default_rng(43)
    V = 20
    bufs = [rng.integers(0, V, 100).astype(np.int32) for _ in range(2)]
    tokens, tok_off = _layout(bufs)
    idx, t_total = build_index(tokens, tok_off, V)
    status = torch.full((2,), -1, dtype=torch.int32, device="cuda")
    seen = []
    for n in (3000, 2000, 7):
        bufs = [np.concatenate([bufs[0], np.full(n, 7, np.int32)]), _grow(rng, bufs[1], 5, V, 0.5)]
        tokens, tok_off = _layout(bufs)
        rs.rs_match_index_append(_cuda(tokens), _cuda(tok_off), 2, V, t_total, idx, status)
        torch.cuda.synchronize()
        seen.append(status.cpu().numpy().copy())
        scores = rng.random(len(tokens)).astype(np.float32)
        for k in (1, 2, 3):
            compare(tokens, tok_off, np.array([k, k], np.int32), None, scores, 0.3, 3, 8, 300, V, idx=idx,
                    t_total=t_total)
    assert seen[0][0] == 0 and seen[1][0] == rs.RS_ST_TRUNCATED and seen[2][0] == rs.RS_ST_TRUNCATED
    assert (np.array(seen)[:, 1] == 0).all()
    # a fresh build holds everything again
    compare(tokens, tok_off, np.array([2, 3], np.int32), None, scores, 0.3, 3, 8, 300, V)
