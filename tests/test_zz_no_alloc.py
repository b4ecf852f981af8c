"""The allocation-free entropy gate, for callers that cannot allocate device
memory (their scratch comes from a fixed array inside the library instead of a
caller workspace).  Checked through the C ABI against rs_entropy_gate on two
calls in a row, each call on fresh logits and carrying the history state
forward, plus its size limit.  Named to be collected last."""
import numpy as np
import pytest
import torch

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


def test_noalloc_gate_matches_workspace_gate_on_two_calls():
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
        o = out["ws"]
        rs.rs_entropy_gate(logits, R, V, row_off, commit, B, p, hist["ws"], hist_n["ws"], o["entropy"],
                           o["k_star"], o["h_best"], o["ok"], ws)
        o = out["na"]
        rs.rs_entropy_gate_noalloc(logits, R, V, row_off, commit, B, p, hist["na"], hist_n["na"],
                                   o["entropy"], o["k_star"], o["h_best"], o["ok"])
        torch.cuda.synchronize()
        a, b = out["ws"], out["na"]
        assert np.abs(host(a["entropy"]) - host(b["entropy"])).max() <= ENT_TOL
        for key in ("k_star", "h_best", "ok"):
            assert (host(a[key]) == host(b[key])).all(), key
        assert (host(hist["ws"]) == host(hist["na"])).all()
        assert (host(hist_n["ws"]) == host(hist_n["na"])).all()


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
