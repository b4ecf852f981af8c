"""The allocation-free entropy gate, for callers that cannot allocate device
memory (their scratch comes from a fixed array inside the library instead of a
caller workspace).  Checked through the C ABI against rs_entropy_gate and the
oracle on two calls in a row, each call on fresh logits and carrying the
history state forward, plus its size limit.  Named to be collected last."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_helpers import ENT_TOL, host
from paper_2511_01282_gb300 import respec as rs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _safe(h_best, hist, hist_n, s):
    """Requests whose trigger a 1e-3 nats entropy error cannot flip: the best
    mean is more than 1e-3 from the threshold and the two best C_k differ by
    more than 1e-3."""
    safe = np.abs(h_best - np.float32(s.theta_entropy)) > 1e-3
    for b in range(len(hist_n)):
        n = int(hist_n[b])
        ck = sorted(hist[b][n - k:n].astype(np.float64).mean() + np.float32(s.lambda_e) / k
                    for k in range(1, n + 1))
        if len(ck) > 1 and ck[1] - ck[0] <= 1e-3:
            safe[b] = False
    return safe


def test_noalloc_gate_matches_workspace_gate_on_two_calls():
    # rs_entropy_gate_noalloc computes the row entropies by the chunked row
    # pass and rs_entropy_gate by the streaming one (when the logits are
    # 16-byte aligned): equal within the entropy tolerance, and each side's
    # trigger is exactly the oracle's trigger on its own entropies
    p = rs.params(l=3)
    # two different batches (different row counts and logits), same requests
    w1 = synth.build(synth.small_spec(B=5, V=20000), seed=31)
    w2 = synth.build(synth.small_spec(B=5, V=20000), seed=32)
    B = w1.B
    hist = {k: _cuda(w1.hist.astype(np.float32)) for k in ("ws", "na")}
    hist_n = {k: _cuda(w1.hist_n.astype(np.int32)) for k in ("ws", "na")}
    for w in (w1, w2):
        R, V = w.logits.shape
        logits = _cuda(w.logits)
        row_off = _cuda(w.node_off.astype(np.int32))
        commit = _cuda(w.row_commit)
        ws = torch.empty(rs.rs_entropy_gate_workspace_size(R, V), dtype=torch.uint8, device="cuda")
        out = {k: dict(entropy=torch.full((R,), -1.0, device="cuda"),
                       k_star=torch.full((B,), -1, dtype=torch.int32, device="cuda"),
                       h_best=torch.full((B,), -1.0, device="cuda"),
                       ok=torch.full((B,), 7, dtype=torch.uint8, device="cuda")) for k in ("ws", "na")}
        before = {k: (host(hist[k]).astype(np.float64), host(hist_n[k])) for k in ("ws", "na")}
        o = out["ws"]
        rs.rs_entropy_gate(logits, R, V, row_off, commit, B, p, hist["ws"], hist_n["ws"], o["entropy"],
                           o["k_star"], o["h_best"], o["ok"], ws)
        o = out["na"]
        rs.rs_entropy_gate_noalloc(logits, R, V, row_off, commit, B, p, hist["na"], hist_n["na"],
                                   o["entropy"], o["k_star"], o["h_best"], o["ok"])
        torch.cuda.synchronize()
        a, b = out["ws"], out["na"]
        H = oracle.entropy_rows(w.logits)
        assert np.abs(host(b["entropy"]) - H).max() <= ENT_TOL
        assert np.abs(host(a["entropy"]) - host(b["entropy"])).max() <= ENT_TOL
        assert (host(hist_n["ws"]) == host(hist_n["na"])).all()
        assert np.abs(host(hist["ws"]) - host(hist["na"])).max() <= ENT_TOL
        hb_a, hb_b = host(a["h_best"]), host(b["h_best"])
        fin = np.isfinite(hb_a)
        assert (np.isfinite(hb_b) == fin).all() and np.abs(hb_a[fin] - hb_b[fin]).max(initial=0) <= ENT_TOL
        for k in ("ws", "na"):  # each trigger: the oracle's, on that side's own entropies
            H_own = host(out[k]["entropy"]).astype(np.float64)
            g = oracle.gate(H_own, w.node_off, w.row_commit, before[k][0], before[k][1], p.l,
                            float(np.float32(p.lambda_e)), float(np.float32(p.theta_entropy)))
            assert (host(out[k]["k_star"]) == g["k_star"]).all(), k
            assert (host(out[k]["ok"]) == g["ok"]).all(), k
            assert (host(out[k]["h_best"]) == g["h_best"].astype(np.float32)).all(), k
            assert (host(hist[k]) == g["hist"].astype(np.float32)).all(), k
        safe = _safe(hb_b, host(hist["na"]), host(hist_n["na"]), p)
        for key in ("k_star", "ok"):  # equal wherever no margin is thin
            assert (host(a[key])[safe] == host(b[key])[safe]).all(), key


def test_noalloc_gate_rejects_oversized_calls():
    p = rs.params(l=3)
    V = 128256                        # 16 chunks of 8192 logits per row
    R = rs.RS_GATE_NOALLOC_MAX_PARTIALS // 16 + 1
    dummy = torch.zeros(1, device="cuda")
    n0 = rs.rs_launch_count()
    with pytest.raises(rs.RespecError) as e:
        rs.rs_entropy_gate_noalloc(dummy, R, V, dummy, dummy, 1, p, dummy, dummy, dummy, dummy,
                                   dummy, dummy)
    assert e.value.status == rs.RS_ERR_CAPACITY
    assert "4096 rows" in str(e.value)
    assert rs.rs_launch_count() == n0
