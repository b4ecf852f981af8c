"""GPU edge cases: malformed and oversized trees, empty requests, unaligned
and odd-sized logits, position-list truncation, skipped requests, and a
CUDA-graph replay of the whole step."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_helpers import check_accept, check_gate, f32, host, make_step
from paper_2511_01282_gb300 import respec as rs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _attn_inputs(rng, Hq, Hkv, D, S_list, trees):
    node_off = np.concatenate([[0], np.cumsum([len(t) for t in trees])]).astype(np.int32)
    sizes = [s + len(t) for s, t in zip(S_list, trees)]
    kv_off = np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)
    T, R = int(sum(sizes)), int(node_off[-1])
    q = synth.bf16_bits(rng.standard_normal((R, Hq, D)).astype(np.float32))
    k = synth.bf16_bits(rng.standard_normal((max(T, 1), Hkv, D)).astype(np.float32))
    v = synth.bf16_bits(rng.standard_normal((max(T, 1), Hkv, D)).astype(np.float32))
    parents = np.concatenate([np.array(t, np.int32) for t in trees]) if R else np.zeros(0, np.int32)
    return q, k, v, kv_off, np.array(S_list, np.int32), node_off, parents


def _run_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, scale):
    B, R = len(ctx), int(node_off[-1])
    out = torch.full((max(R, 1), Hq, D), 7.0, device="cuda")
    lse = torch.full((max(R, 1), Hq), 7.0, device="cuda")
    status = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    ws = torch.empty(rs.rs_tree_verify_attn_workspace_size(B, R, Hq, Hkv, D), dtype=torch.uint8, device="cuda")
    rs.rs_tree_verify_attn(_cuda(q), _cuda(k), _cuda(v), k.shape[0], _cuda(kv_off), _cuda(ctx), _cuda(node_off),
                           _cuda(parents) if R else None, B, R, Hq, Hkv, D, scale, out, lse, status, ws)
    torch.cuda.synchronize()
    return host(out)[:R], host(lse)[:R], host(status)


def test_attention_rejects_bad_trees_and_keeps_the_rest():
    rng = np.random.default_rng(0)
    Hq, Hkv, D = 4, 2, 128
    good = [-1, 0, 0, 1, 3]
    trees = [good, [-1, 0, 2, 1], [], [-1] + [int(rng.integers(0, i)) for i in range(1, 300)], good]
    S = [130, 50, 10, 200, 0]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert status.tolist() == [0, rs.RS_ST_BAD_TREE, 0, rs.RS_ST_TOO_LARGE, 0]
    q, k, v, kv_off, ctx, node_off, parents = inp
    for b in (1, 3):
        n0, n1 = node_off[b], node_off[b + 1]
        assert (out[n0:n1] == 0).all() and (lse[n0:n1] == 0).all()
    for b in (0, 4):  # S = 0 for request 4: the tree alone
        n0, n1 = int(node_off[b]), int(node_off[b + 1])
        rows = [(n, h) for n in range(n0, n1) for h in range(Hq)]
        ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5, rows=rows)
        got = out[n0:n1].reshape(-1, D)
        assert np.abs(got - ref["out"]).max() < 1e-2


@pytest.mark.parametrize("B,ctx_hi,D", [(3840, 12, 64), (300, 400, 128)])
def test_attention_many_requests(B, ctx_hi, D):
    # the largest request count a call takes (two prefixes over the requests
    # in shared memory), and a few hundred short requests whose segments the
    # cost-weighted split spreads over the CTAs (some ranges empty)
    rng = np.random.default_rng(B)
    Hq, Hkv = 2, 1
    trees = []
    for _ in range(B):
        n = int(rng.integers(1, 6))
        trees.append([-1] + [int(rng.integers(0, i)) for i in range(1, n)])
    S = [int(x) for x in rng.integers(0, ctx_hi, B)]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert (status == 0).all()
    q, k, v, kv_off, ctx, node_off, parents = inp
    R = int(node_off[-1])
    rows = [(n, h) for n in range(0, R, max(1, R // 600)) for h in range(Hq)]
    ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5, rows=rows)
    got = np.stack([out[n, h] for n, h in rows])
    assert np.abs(got - ref["out"].reshape(len(rows), D)).max() < 1e-2


def test_attention_wait_time_out_reports_status_and_recovers(monkeypatch):
    # every pipeline wait limited to 200 clock cycles: the first waits give
    # up, the CTAs drain their copies and MMAs, free TMEM and flag the
    # requests they held; the next call, with the normal limit, is correct
    rng = np.random.default_rng(2)
    Hq, Hkv, D = 4, 2, 128
    trees = [[-1, 0, 0, 1], [-1] + [int(rng.integers(0, i)) for i in range(1, 40)]]
    S = [700, 1500]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    monkeypatch.setenv("RS_DEBUG_WAIT_LIMIT", "200")
    _, _, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert (status & rs.RS_ST_TIMEOUT).any()
    monkeypatch.delenv("RS_DEBUG_WAIT_LIMIT")
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert (status == 0).all()
    q, k, v, kv_off, ctx, node_off, parents = inp
    ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5)
    assert np.abs(out.reshape(-1, D) - ref["out"]).max() < 1e-2


def test_attention_single_node_and_tile_straddling_tree():
    rng = np.random.default_rng(1)
    Hq, Hkv, D = 6, 3, 64
    trees = [[-1], [-1] + list(range(0, 99)), [-1, 0, 1, 1, 0]]
    S = [1, 90, 127]  # tree slots cross the 128-key tile boundary
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, 0.3)
    assert (status == 0).all()
    q, k, v, kv_off, ctx, node_off, parents = inp
    ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, 0.3)
    assert np.abs(out.reshape(-1, D) - ref["out"]).max() < 1e-2
    assert np.abs(lse.reshape(-1) - ref["lse"]).max() < 1e-3


def test_accept_rejects_bad_trees():
    w = synth.build(synth.small_spec(B=4, V=700), seed=11)
    # request 2: a model node hanging from a chain node
    n0 = int(w.node_off[2])
    src = w.source.copy()
    ch = w.chain.copy()
    src[n0 + 1], ch[n0 + 1] = 2, 0
    w.source, w.chain = src, ch
    st = make_step(w)
    ref = check_accept(w, st)
    assert ref["status"][2] & oracle.ST_BAD_TREE


def test_unaligned_and_odd_logits():
    w = synth.build(synth.small_spec(B=2, V=1003), seed=12)
    st = make_step(w)
    R, V = w.logits.shape
    flat = torch.zeros(R * V + 1, dtype=torch.float32, device="cuda")
    flat[1:] = torch.from_numpy(w.logits.reshape(-1)).cuda()
    st.d["logits"] = flat[1:].view(R, V)  # 4-byte aligned only: scalar path
    check_gate(w, st)
    check_accept(w, st)


@pytest.mark.parametrize("V,beta", [(8193, 5), (20003, 16), (65536, 16), (65537, 16), (70000, 5),
                                    (100000, 16), (131072, 5), (131073, 5)])
def test_accept_chunk_counts(V, beta):
    # rows of 2 to 8 chunks of 8192 logits are merged inside their cluster,
    # longer rows (9 to 17 chunks here) by the separate merge kernel, up to
    # its 256 candidates a row; V % 4 != 0 takes scalar loads
    w = synth.build(synth.small_spec(B=2, V=V, beta=beta), seed=V % 97)
    st = make_step(w)
    check_accept(w, st)


@pytest.mark.parametrize("V,B,beta,nodes", [(8, 3, 4, (1, 4)), (1024, 2, 5, (20, 40)), (4096, 2, 16, (20, 40)),
                                               (4100, 3, 5, (20, 40)), (32000, 12, 5, (20, 40)),
                                               (12288, 24, 16, (20, 40))])
def test_logits_row_pass_sizes(V, B, beta, nodes):
    # the gate and accept row passes on rows far shorter than one 8192-logit
    # chunk, of exactly half and a little over half of one, and with more rows
    # (B = 12, 24) than the GPU has SMs
    w = synth.build(synth.small_spec(B=B, V=V, beta=beta, model_nodes=nodes), seed=V % 89 + B)
    st = make_step(w)
    check_gate(w, st)
    check_accept(w, st)


def test_logits_row_pass_masked_rows():
    # rows with only a few finite logits (the rest -inf), fewer than beta in
    # some: the top-beta list keeps -inf entries in id order, as the oracle
    w = synth.build(synth.small_spec(B=3, V=6000, beta=8), seed=16)
    rng = np.random.default_rng(16)
    z = w.logits.copy()
    for r in range(z.shape[0]):
        keep = rng.choice(z.shape[1], size=int(rng.integers(1, 12)), replace=False)
        mask = np.ones(z.shape[1], bool)
        mask[keep] = False
        if r % 3 == 0:  # also keep the row's draft children finite
            mask[w.tree_tokens[w.node_off[0]:w.node_off[-1]]] = False
        z[r, mask] = -np.inf
    w.logits = z
    st = make_step(w)
    check_gate(w, st)
    check_accept(w, st)


def test_accept_without_entropy_output():
    w = synth.build(synth.small_spec(B=3, V=5000), seed=15)
    st = make_step(w)
    st.out["acc_entropy"].fill_(-5.0)
    st.accept(entropy=False)
    torch.cuda.synchronize()
    assert (host(st.out["acc_entropy"]) == -5.0).all()  # untouched
    st.d["scores"].copy_(torch.from_numpy(w.scores))
    check_accept(w, st)


def test_scan_truncation_and_skips():
    w = synth.build(synth.small_spec(B=4, repeat_prob=0.9, seg_len=(2, 4), V=50), seed=13)
    st = make_step(w)
    st.pos_cap = 3
    st.out["pos"] = torch.zeros((w.B, 3), dtype=torch.int32, device="cuda")
    ks = np.array([1, 2, 9, 3], np.int32)          # 9 > RS_MAX_L: skipped with a status
    ok = np.array([1, 1, 1, 0], np.uint8)          # request 3 not triggered
    ks_o = ks.copy()
    ks_o[2] = 0
    # the oracle has no key-length cap: it sees the capped request as k = 0
    st.scan(k_star=_cuda(ks), gate_ok=_cuda(ok))
    torch.cuda.synchronize()
    ref = oracle.match_scan(w.tokens, w.tok_off, ks_o, w.scores, f32(w.spec.theta_score), w.spec.top_c,
                            w.spec.chain_len, 3, gate_ok=ok)
    got_status = host(st.out["scan_status"])
    assert got_status[2] == rs.RS_ST_TOO_LARGE
    for key in ("count", "pos", "sel_pos", "sel_len", "spans", "n_sel"):
        assert (host(st.out[key]) == ref[key]).all(), key
    assert got_status[0] & rs.RS_ST_TRUNCATED and got_status[3] == 0
    assert (ref["status"][[0, 1, 3]] == got_status[[0, 1, 3]]).all()


def test_gate_with_empty_row_ranges():
    w = synth.build(synth.small_spec(B=3, V=300), seed=14)
    st = make_step(w)
    # request 1 owns no rows this step: its history is only re-evaluated
    off = w.node_off.copy()
    off[2] = off[1]
    st.d["row_off"] = _cuda(off.astype(np.int32))
    st.gate()
    torch.cuda.synchronize()
    H = host(st.out["entropy"]).astype(np.float64)
    g = oracle.gate(H, off, w.row_commit, w.hist, w.hist_n, w.spec.l, f32(w.spec.lambda_e),
                    f32(w.spec.theta_entropy))
    assert (host(st.out["k_star"]) == g["k_star"]).all()
    assert (host(st.d["hist"]) == g["hist"].astype(np.float32)).all()


def test_cuda_graph_replay_matches_eager():
    # the fused step (trigger on the previous accept's row entropies) and the
    # unfused one, each captured once and replayed: same outputs as eager
    w = synth.make("tiny")
    for fused in (True, False):
        st = make_step(w)
        st.prime()
        torch.cuda.synchronize()
        carried = st.out["acc_entropy"].clone()  # the fused trigger's input
        st.step(fused=fused)
        torch.cuda.synchronize()
        skip = {"acc_entropy"} | ({"entropy"} if fused else set())
        eager = {k: host(v).copy() for k, v in st.out.items() if k not in skip}

        def reset():
            st.reset_state()
            st.out["acc_entropy"].copy_(carried)

        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        reset()
        torch.cuda.synchronize()
        with torch.cuda.stream(s):
            st.step(stream=s, fused=fused)  # warm the stream once outside the capture
        torch.cuda.synchronize()
        reset()
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=s):
            st.step(stream=s, fused=fused)
        reset()
        for k in eager:
            st.out[k].fill_(-3)  # the replay has to rewrite every output
        torch.cuda.synchronize()
        n0 = rs.rs_launch_count()
        with torch.cuda.stream(s):
            g.replay()
        torch.cuda.synchronize()
        assert rs.rs_launch_count() == n0  # replays do not go through the host entry points
        for k, v in eager.items():
            assert (host(st.out[k]) == v).all(), (fused, k)


def _scan_direct(tokens, tok_off, ks, ok, scores, theta, top_c, span_len, pos_cap):
    B = len(tok_off) - 1
    z = lambda *shape: torch.full(shape, -7, dtype=torch.int32, device="cuda")  # noqa: E731
    out = dict(count=z(B), pos=z(B, pos_cap), sel_pos=z(B, top_c), sel_len=z(B, top_c),
               spans=z(B, top_c, span_len), n_sel=z(B), status=z(B))
    p = rs.params(theta_score=theta, top_c=top_c, span_len=span_len)
    rs.rs_match_scan(_cuda(tokens), _cuda(tok_off), B, _cuda(ks), _cuda(ok), _cuda(scores), p, pos_cap,
                     out["count"], out["pos"], out["sel_pos"], out["sel_len"], out["spans"], out["n_sel"],
                     out["status"])
    torch.cuda.synchronize()
    return {k: host(v) for k, v in out.items()}


@pytest.mark.parametrize("dense", [False, True])
def test_scan_long_buffers(dense):
    # buffer lengths at the one-CTA limit (8192), just above it (split over the
    # cluster, one window per CTA), at the one-window-per-CTA limit (65537) and
    # well past it (several windows per CTA); dense: a 3-token vocabulary, so
    # thousands of matches overflow the shared candidate buffer and pos_cap
    rng = np.random.default_rng(21 + dense)
    lens = [8192, 8193, 65537, 65538, 150001]
    V = 3 if dense else 200
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tokens = rng.integers(0, V, int(tok_off[-1])).astype(np.int32)
    for b, t in enumerate(lens):  # plant the key earlier so sparse buffers match too
        a = int(tok_off[b])
        for q in rng.integers(8, t - 8, 6):
            tokens[a + q - 3:a + q + 1] = tokens[a + t - 4:a + t]
    scores = rng.random(int(tok_off[-1])).astype(np.float32)
    scores[rng.random(scores.size) < 0.1] = 0.75  # ties on the score
    ks = np.array([1, 2, 3, 4, 2], np.int32)
    ok = np.ones(len(lens), np.uint8)
    theta, top_c, span_len, pos_cap = 0.3, 8, 16, 5000
    got = _scan_direct(tokens, tok_off, ks, ok, scores, theta, top_c, span_len, pos_cap)
    ref = oracle.match_scan(tokens, tok_off, ks, scores, f32(theta), top_c, span_len, pos_cap, gate_ok=ok)
    for key in ("count", "pos", "sel_pos", "sel_len", "spans", "n_sel", "status"):
        assert (got[key] == ref[key]).all(), key
    assert (ref["n_sel"] > 0).all()


# ------------------------------------------------------------------ offsets out of bounds
# Offsets arrays are device data the host cannot check: every kernel checks the
# ranges it reads before indexing with them.  Requests 1 and 2 get ranges that
# run past the arrays (past R, kv_rows or the buffers' tok_off[B] tokens, or a
# negative length); they are reported RS_ST_BAD_OFFSET and skipped, and
# request 0 (same range as in the valid workload) still matches the oracle.
BIG = 1 << 28


def _bad_offsets(off):
    """off[B+1] with request 1's end and request 2's start far past the end."""
    bad = np.array(off, dtype=np.int64).copy()
    bad[2] = BIG
    return bad


def test_attention_offsets_out_of_bounds():
    w = synth.build(synth.small_spec(B=3, V=500), seed=21)
    s = w.spec
    st = make_step(w)
    node_off = _bad_offsets(w.node_off).astype(np.int32)
    st.d["node_off"] = _cuda(node_off)
    st.attn()
    torch.cuda.synchronize()
    status = host(st.out["attn_status"])
    assert status[0] == 0 and status[1] == rs.RS_ST_BAD_OFFSET and status[2] == rs.RS_ST_BAD_OFFSET
    n0, n1 = int(w.node_off[0]), int(w.node_off[1])
    rows = [(n, h) for n in range(n0, n1) for h in range(s.Hq)]
    ref = oracle.tree_attn(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents, s.Hq, s.Hkv, s.D,
                           st.scale, rows=rows)
    got = host(st.out["attn_out"])[n0:n1].reshape(-1, s.D)
    assert np.abs(got - ref["out"]).max() < 1e-2
    # keys past kv_rows: request 2's prefix ends beyond the KV cache
    st = make_step(w)
    kv_off = w.kv_off.copy()
    kv_off[2] = st.kv_rows - 1
    st.d["kv_off"] = _cuda(kv_off)
    st.attn()
    torch.cuda.synchronize()
    assert host(st.out["attn_status"]).tolist() == [0, 0, rs.RS_ST_BAD_OFFSET]


def test_accept_and_sample_offsets_out_of_bounds():
    w = synth.build(synth.small_spec(B=3, V=700), seed=22)
    s = w.spec
    ref = oracle.accept(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, w.chain, w.sel_pos,
                        w.tok_off, w.scores, s.beta, f32(s.tau), s.phi, s.m, f32(s.alpha), 64)
    st = make_step(w)
    st.d["node_off"] = _cuda(_bad_offsets(w.node_off).astype(np.int32))
    st.accept()
    torch.cuda.synchronize()
    o = st.out
    stt = host(o["acc_status"])
    assert stt[0] == ref["status"][0] and stt[1] == rs.RS_ST_BAD_OFFSET and stt[2] == rs.RS_ST_BAD_OFFSET
    for k in ("acc_len", "bonus", "winner"):
        assert host(o[k])[0] == ref[k][0], k
    assert (host(o["acc_nodes"])[0] == ref["acc_nodes"][0]).all()
    assert (host(o["winner"])[1:] == -2).all() and (host(o["acc_len"])[1:] == 0).all()
    # the score table: request 0's selected positions updated as the oracle's, the rest untouched
    t1 = int(w.tok_off[1])
    assert (host(st.d["scores"])[:t1] == ref["scores"][:t1]).all()
    assert (host(st.d["scores"])[t1:] == w.scores[t1:]).all()
    # tok_off past the score table for request 1
    st = make_step(w)
    tok_off = w.tok_off.copy()
    tok_off[2] = tok_off[3] + 5
    st.d["tok_off"] = _cuda(tok_off)
    st.accept()
    torch.cuda.synchronize()
    assert host(st.out["acc_status"])[1] & rs.RS_ST_BAD_OFFSET
    # sampling walk
    st = make_step(w)
    st.d["node_off"] = _cuda(_bad_offsets(w.node_off).astype(np.int32))
    st.tree_sample(1.0)
    torch.cuda.synchronize()
    so = {k: host(v) for k, v in st.sample_out.items()}
    assert so["status"][1] == rs.RS_ST_BAD_OFFSET and so["status"][2] == rs.RS_ST_BAD_OFFSET
    assert so["acc_len"][1] == 0 and so["bonus"][1] == -1


def test_scan_gate_and_index_offsets_out_of_bounds():
    w = synth.build(synth.small_spec(B=3, V=300, repeat_prob=0.6, seg_len=(3, 8)), seed=23)
    s = w.spec
    ks = np.array([2, 2, 2], np.int32)
    tok_bad = _bad_offsets(w.tok_off)
    tok_bad[-1] = w.tok_off[-1]              # the buffers hold tok_off[B] tokens
    ref = oracle.match_scan(w.tokens, w.tok_off, ks, w.scores, f32(s.theta_score), s.top_c, s.chain_len,
                            s.pos_cap)
    st = make_step(w)
    st.d["tok_off"] = _cuda(tok_bad)
    st.scan(k_star=_cuda(ks), gate_ok=None)
    torch.cuda.synchronize()
    o = st.out
    assert host(o["scan_status"]).tolist()[1:] == [rs.RS_ST_BAD_OFFSET] * 2
    for k_gpu, k_ref in (("count", "count"), ("pos", "pos"), ("sel_pos", "sel_pos"), ("spans", "spans")):
        assert (host(o[k_gpu])[0] == ref[k_ref][0]).all(), k_gpu
    assert (host(o["n_sel"])[1:] == 0).all()
    # the trigger: a request whose rows run past the entropies pushes nothing
    st = make_step(w)
    row_bad = _bad_offsets(w.node_off).astype(np.int32)
    st.d["row_off"] = _cuda(row_bad)
    st.out["acc_entropy"].copy_(torch.from_numpy(oracle.entropy_rows(w.logits).astype(np.float32)))
    st.gate_rows()
    torch.cuda.synchronize()
    H = host(st.out["acc_entropy"]).astype(np.float64)
    off0 = np.array([0, w.node_off[1], w.node_off[1], w.node_off[1]], np.int64)  # rows of request 0 only
    g = oracle.gate(H, off0, w.row_commit, w.hist, w.hist_n, s.l, f32(s.lambda_e), f32(s.theta_entropy))
    assert (host(st.out["k_star"]) == g["k_star"]).all() and (host(st.d["hist"]) == g["hist"].astype(np.float32)).all()
    # the index: a build on inconsistent offsets holds nothing; a query with a
    # request out of bounds skips it
    from test_gpu_index import build_index, query
    idx, t_total = build_index(w.tokens, tok_bad, s.V)
    got = query(w.tokens, w.tok_off, ks, None, w.scores, s.theta_score, s.top_c, s.chain_len, 16, s.V, t_total, idx)
    assert (got["status"] == rs.RS_ST_BAD_OFFSET).all()
    status = torch.zeros(3, dtype=torch.int32, device="cuda")
    rs.rs_match_index_append(_cuda(w.tokens), _cuda(w.tok_off), 3, s.V, t_total, idx, status)
    torch.cuda.synchronize()
    assert (host(status) == rs.RS_ST_BAD_OFFSET).all()
    idx, t_total = build_index(w.tokens, w.tok_off, s.V)
    got = query(w.tokens, tok_bad, ks, None, w.scores, s.theta_score, s.top_c, s.chain_len, 16, s.V, t_total, idx)
    ref16 = oracle.match_scan(w.tokens, w.tok_off, ks, w.scores, f32(s.theta_score), s.top_c, s.chain_len, 16)
    assert got["status"].tolist()[1:] == [rs.RS_ST_BAD_OFFSET] * 2
    for k in ("count", "pos", "sel_pos", "spans"):
        assert (got[k][0] == ref16[k][0]).all(), k
