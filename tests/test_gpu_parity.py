"""GPU parity: every C-ABI call against the oracle on the same seeded inputs.

Full oracle comparison on every workload: the tiny and 7B-shape workloads,
ragged small workloads (several KV tiles, ragged tails, GQA groups 1-8, head
dims 64 and 128) and the long-context and batched full sizes in the launch
configuration the benchmark times (the attention oracle fanned out over host
threads by row chunks).
"""
import numpy as np
import pytest
import torch

import synth
from gpu_helpers import check_accept, check_attn, check_gate, check_gate_rows, check_scan, make_step

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available()


def _all_checks(w, attn_rows=None):
    st = make_step(w)
    g = check_gate(w, st)
    check_scan(w, st)                                   # explicit key lengths
    check_scan(w, st, k_star=g["k_star"], gate_ok=g["ok"])  # keyed and gated by the trigger
    check_attn(w, st, rows=attn_rows)
    check_accept(w, st)
    check_gate_rows(w, st)                                  # trigger on rs_accept's entropies
    return st


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_named_config_full(name):
    _all_checks(synth.make(name))


SMALL = [
    dict(seed=1),
    dict(seed=2, Hq=4, Hkv=4, D=64, ctx=(0, 300)),
    dict(seed=3, Hq=20, Hkv=4, D=128, ctx=(120, 140), model_nodes=(60, 120), n_chains=(2, 3)),
    dict(seed=4, B=5, Hq=8, Hkv=8, D=64, V=1001, ctx=(1, 1000), beta=16, top_c=8, n_chains=(3, 8),
         chain_len=9, l=5),
    dict(seed=5, B=2, Hq=16, Hkv=2, D=128, V=4096, ctx=(2000, 2600), model_nodes=(200, 240),
         max_depth=12, n_chains=(1, 3), chain_len=12, tau=0.5, m=1, phi=3),
    dict(seed=6, B=7, Hq=8, Hkv=1, D=128, V=512, ctx=(5, 400), model_nodes=(1, 6), n_chains=(0, 1),
         chain_len=3, repeat_prob=0.6, seg_len=(2, 6), score_noise=0.6, theta_score=0.45),
    # D = 64 with two or three 128-row tiles per KV head and enough KV tiles
    # that every CTA's range is non-empty: split segments of several pieces
    dict(seed=7, B=3, Hq=8, Hkv=4, D=64, V=2048, ctx=(1500, 2500), model_nodes=(80, 120), max_depth=8,
         n_chains=(1, 3), chain_len=8),
]


@pytest.mark.parametrize("kw", SMALL, ids=[str(i) for i in range(len(SMALL))])
def test_small_ragged_full(kw):
    kw = dict(kw)
    seed = kw.pop("seed")
    _all_checks(synth.build(synth.small_spec(**kw), seed=seed))


@pytest.mark.slow
@pytest.mark.parametrize("name", ["gqa16k", "batched", "13b32k"])
def test_full_size_configs(name):
    # every (node, head) row of the attention, every row and request of the rest
    w = synth.make(name)
    _all_checks(w, attn_rows=None)


def test_repeated_steps_carry_state():
    # two gate + accept rounds: history and scores evolve exactly as the oracle's
    import oracle
    from gpu_helpers import f32, host
    w = synth.build(synth.small_spec(B=3, V=2000), seed=9)
    s = w.spec
    st = make_step(w)
    hist, hist_n, scores = w.hist.astype(np.float64), w.hist_n, w.scores
    for _ in range(2):
        st.gate()
        st.accept()
        torch.cuda.synchronize()
        H = host(st.out["entropy"]).astype(np.float64)
        g = oracle.gate(H, w.node_off, w.row_commit, hist, hist_n, s.l, f32(s.lambda_e), f32(s.theta_entropy))
        hist, hist_n = g["hist"], g["hist_n"]
        a = oracle.accept(w.logits, w.node_off, w.tree_tokens, w.parents, w.source, w.chain, w.sel_pos,
                          w.tok_off, scores, s.beta, f32(s.tau), s.phi, s.m, f32(s.alpha), st.acc_cap)
        scores = a["scores"]
        assert (host(st.d["hist"]) == hist.astype(np.float32)).all()
        assert (host(st.d["scores"]) == scores).all()
        assert (host(st.out["commit"]) == a["commit"]).all()
