"""Shared parity checks: run the C-ABI calls on the GPU and compare each
output with the oracle on the same seeded inputs.

Tolerances, per output (exact where the result is an integer or a decision,
the arithmetic's rounding bound otherwise):
  * match positions, counts, spans, selections, argmax, top-beta ids,
    acceptance decisions, accepted paths, winners, bonus tokens, commit flags,
    status words and updated scores: bit-exact;
  * row entropy: 1e-3 nats (fp32 accumulation vs fp64);
  * attention output: max |err| <= 1e-2 and relative L2 <= 1e-2 (bf16 inputs,
    fp32 accumulation);
  * log-sum-exp: 1e-5 relative (fp32 exp/log); token probability
    p = exp(z - lse): 1e-5 * max(1, |lse|) relative, the lse bound carried
    through the exponential.
Where floating point decides an integer (the trigger's k* near a tie or the
threshold), the oracle takes the decision on the GPU's own fp32 entropies.
"""
import numpy as np
import torch

import oracle
from paper_2511_01282_gb300 import respec as rs
from paper_2511_01282_gb300.pipeline import VerifyStep, arrays_from_workload

ENT_TOL = 1e-3
ATTN_MAX_ABS = 1e-2
ATTN_REL_L2 = 1e-2
LSE_REL = 1e-5


def f32(x):
    return float(np.float32(x))


def make_step(w, **kw):
    s = w.spec
    p = rs.params(**s.params())
    return VerifyStep(arrays_from_workload(w), p, s.Hq, s.Hkv, s.D, pos_cap=s.pos_cap, **kw)


def host(t):
    return t.detach().cpu().numpy()


# ------------------------------------------------------------------ gate
def check_gate(w, st):
    s = w.spec
    st.gate()
    torch.cuda.synchronize()
    o = st.out
    H = oracle.entropy_rows(w.logits)
    got = host(o["entropy"]).astype(np.float64)
    err = np.max(np.abs(got - H)) if H.size else 0.0
    assert err <= ENT_TOL, "entropy error %g nats" % err
    # trigger on the GPU's entropies: bit-exact
    g = oracle.gate(got, w.node_off, w.row_commit, w.hist, w.hist_n, s.l, f32(s.lambda_e),
                    f32(s.theta_entropy))
    assert (host(o["k_star"]) == g["k_star"]).all()
    assert (host(o["entropy_ok"]) == g["ok"]).all()
    assert (host(o["h_best"]) == g["h_best"].astype(np.float32)).all()
    assert (host(st.d["hist_n"]) == g["hist_n"]).all()
    assert (host(st.d["hist"]) == g["hist"].astype(np.float32)).all()
    # trigger on the oracle's own entropies: equal wherever no margin is thin
    g2 = oracle.gate(H, w.node_off, w.row_commit, w.hist, w.hist_n, s.l, f32(s.lambda_e),
                     f32(s.theta_entropy))
    safe = np.abs(g2["h_best"] - f32(s.theta_entropy)) > 1e-3
    for b in range(w.B):  # thin C_k margins may flip k* under a 1e-3 entropy error
        n = int(g2["hist_n"][b])
        hb = g2["hist"][b][:n]
        ck = sorted(hb[n - k:].mean() + f32(s.lambda_e) / k for k in range(1, n + 1))
        if len(ck) > 1 and ck[1] - ck[0] <= 1e-3:
            safe[b] = False
    assert (host(o["k_star"])[safe] == g2["k_star"][safe]).all()
    assert (host(o["entropy_ok"])[safe] == g2["ok"][safe]).all()
    return g


# ------------------------------------------------------------------ scan
def check_scan(w, st, k_star=None, gate_ok=None, pos_cap=None):
    s = w.spec
    ks = w.k_star_hint if k_star is None else k_star
    kd = torch.from_numpy(np.ascontiguousarray(ks, np.int32)).cuda()
    okd = None if gate_ok is None else torch.from_numpy(np.ascontiguousarray(gate_ok, np.uint8)).cuda()
    st.scan(k_star=kd, gate_ok=okd)
    torch.cuda.synchronize()
    o = st.out
    ref = oracle.match_scan(w.tokens, w.tok_off, ks, w.scores, f32(s.theta_score), s.top_c,
                            s.chain_len, st.pos_cap, gate_ok=gate_ok)
    for k_gpu, k_ref in (("count", "count"), ("pos", "pos"), ("sel_pos", "sel_pos"),
                         ("sel_len", "sel_len"), ("spans", "spans"), ("n_sel", "n_sel"),
                         ("scan_status", "status")):
        a, b = host(o[k_gpu]), ref[k_ref]
        assert a.shape == b.shape and (a == b).all(), "scan %s differs" % k_gpu
    return ref


# ------------------------------------------------------------------ attention
def oracle_attn(w, scale, rows=None, workers=None):
    """oracle.tree_attn over (node, head) rows (every row when None), split
    into disjoint chunks that host threads run at once.  The oracle's C code
    runs with the GIL released and computes each row on its own, so the
    split changes nothing in its arithmetic; it only makes the full-size
    comparison take seconds instead of minutes."""
    import concurrent.futures as cf
    import os
    s = w.spec
    if rows is None:
        rr = np.stack(np.meshgrid(np.arange(w.R), np.arange(s.Hq), indexing="ij"), -1).reshape(-1, 2)
    else:
        rr = np.asarray(list(rows), dtype=np.int64).reshape(-1, 2)
    nw = max(1, min(workers or os.cpu_count() or 1, 64, len(rr)))
    parts = np.array_split(rr, nw * 4) if len(rr) > 0 else [rr]

    def run(part):
        return oracle.tree_attn(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents, s.Hq, s.Hkv,
                                s.D, scale, rows=part)

    with cf.ThreadPoolExecutor(max_workers=nw) as ex:
        res = list(ex.map(run, parts))
    return dict(out=np.concatenate([r["out"] for r in res]), lse=np.concatenate([r["lse"] for r in res]),
                rows=np.concatenate([r["rows"] for r in res]), rc=max(r["rc"] for r in res))


def check_attn(w, st, rows=None):
    """rs_tree_verify_attn against the oracle on the given (node, head) rows,
    every row when None."""
    st.attn()
    torch.cuda.synchronize()
    o = st.out
    ref = oracle_attn(w, st.scale, rows=rows)
    assert ref["rc"] == 0
    rr = ref["rows"]
    got = host(o["attn_out"])[rr[:, 0], rr[:, 1]].astype(np.float64)
    lse = host(o["attn_lse"])[rr[:, 0], rr[:, 1]].astype(np.float64)
    err = np.abs(got - ref["out"])
    rel = np.linalg.norm(got - ref["out"]) / max(np.linalg.norm(ref["out"]), 1e-30)
    assert err.max() <= ATTN_MAX_ABS, "attention max abs error %g" % err.max()
    assert rel <= ATTN_REL_L2, "attention rel L2 error %g" % rel
    lerr = np.abs(lse - ref["lse"]) / np.maximum(np.abs(ref["lse"]), 1.0)
    assert lerr.max() <= 1e-4, "attention lse error %g" % lerr.max()
    assert (host(o["attn_status"]) == 0).all()
    return err.max(), rel


# ------------------------------------------------------------------ accept
def check_accept(w, st, acc_cap=None):
    s = w.spec
    st.accept()
    torch.cuda.synchronize()
    o = st.out
    ref = oracle.accept(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, w.chain, w.sel_pos,
                        w.tok_off, w.scores, s.beta, f32(s.tau), s.phi, s.m, f32(s.alpha), st.acc_cap)
    for k_gpu, k_ref in (("argmax", "argmax"), ("topk", "topk"), ("acc_len", "acc_len"),
                         ("acc_nodes", "acc_nodes"), ("bonus", "bonus"), ("winner", "winner"),
                         ("commit", "commit"), ("acc_status", "status")):
        a, b = host(o[k_gpu]), ref[k_ref]
        assert a.shape == b.shape and (a == b).all(), "accept %s differs" % k_gpu
    assert (host(st.d["scores"]) == ref["scores"]).all(), "updated scores differ"
    # the row entropies of the same pass (rs_accept's fused output)
    H = oracle.entropy_rows(w.logits)
    err = np.max(np.abs(host(o["acc_entropy"]).astype(np.float64) - H)) if H.size else 0.0
    assert err <= ENT_TOL, "accept entropy error %g nats" % err
    lse = host(o["lse"]).astype(np.float64)
    assert np.allclose(lse, ref["lse"], rtol=LSE_REL, atol=1e-6)
    # p(token) = exp(z - lse(parent row)): an lse within its relative bound
    # LSE_REL moves p by up to LSE_REL * |lse(parent)| relatively
    pt = host(o["p_tok"]).astype(np.float64)
    tol = np.full(pt.shape, LSE_REL)
    for b in range(w.B):
        n0, n1 = int(w.node_off[b]), int(w.node_off[b + 1])
        for i in range(n0 + 1, n1):
            par = n0 + int(w.parents[i])
            if n0 <= par < i:
                tol[i] = LSE_REL * max(1.0, abs(ref["lse"][par]))
    assert (np.abs(pt - ref["p_tok"]) <= tol * ref["p_tok"] + 1e-7).all()
    return ref


# ------------------------------------------------------------------ gate from rows
def check_gate_rows(w, st):
    """rs_entropy_gate_rows on rs_accept's entropies: bit-exact trigger."""
    s = w.spec
    st.d["hist"].copy_(torch.from_numpy(w.hist))
    st.d["hist_n"].copy_(torch.from_numpy(w.hist_n))
    st.gate_rows()
    torch.cuda.synchronize()
    o = st.out
    H = host(o["acc_entropy"]).astype(np.float64)
    g = oracle.gate(H, w.node_off, w.row_commit, w.hist, w.hist_n, s.l, f32(s.lambda_e),
                    f32(s.theta_entropy))
    assert (host(o["k_star"]) == g["k_star"]).all()
    assert (host(o["entropy_ok"]) == g["ok"]).all()
    assert (host(o["h_best"]) == g["h_best"].astype(np.float32)).all()
    assert (host(st.d["hist"]) == g["hist"].astype(np.float32)).all()
    assert (host(st.d["hist_n"]) == g["hist_n"]).all()
