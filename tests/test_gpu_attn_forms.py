"""GPU parity of both forms of rs_tree_verify_attn's main kernel.

The call picks the two-row-tile form (a segment is a pair of 128-row tiles
sharing every K/V tile) when its requests average more than one row tile per
KV head, and the one-tile form otherwise.  RS_DEBUG_ATTN_FORM=one|pair
forces either, so each is checked against the oracle on every (node, head)
row of shapes that exercise its paths: full pairs, half pairs (a request of
one tile, or the last pair of an odd tile count), segments split over
several CTAs, head dims 64 and 128, GQA groups 1-16 (Q tiles copied by
TMA) and 5 (Q tiles written by the softmax threads), masks crossing tiles,
rejected requests, many requests, launches that stream K/V from HBM, and
the bounded-wait time-out.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_helpers import check_attn, host, make_step
from paper_2511_01282_gb300 import respec as rs
from test_gpu_edges import _attn_inputs, _run_attn

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    assert torch.cuda.is_available()


SHAPES = [
    # one request, GQA 8: 1 .. 4 row-tile pairs per KV head, split segments
    dict(seed=21, B=1, Hq=32, Hkv=4, D=128, V=512, ctx=(3000, 3000), model_nodes=(100, 100), n_chains=(2, 2),
         chain_len=8),
    # ragged batch: requests of one tile (half pairs) and of several
    dict(seed=22, B=6, Hq=16, Hkv=2, D=128, V=512, ctx=(1, 2500), model_nodes=(4, 60), n_chains=(0, 3),
         chain_len=6),
    # GQA 16 over 130+ nodes: odd tile counts, last pair half
    dict(seed=23, B=2, Hq=16, Hkv=1, D=128, V=512, ctx=(900, 1400), model_nodes=(120, 140), n_chains=(1, 2),
         chain_len=10),
    # head dim 64, group 4
    dict(seed=24, B=3, Hq=8, Hkv=2, D=64, V=512, ctx=(1500, 2500), model_nodes=(80, 120), max_depth=8,
         n_chains=(1, 3), chain_len=8),
    # no GQA (group 1): every request is one half pair
    dict(seed=25, B=4, Hq=8, Hkv=8, D=128, V=512, ctx=(100, 700), model_nodes=(10, 40), n_chains=(1, 2),
         chain_len=5),
    # group 5 (does not divide 128): the softmax threads write the Q tiles
    dict(seed=26, B=2, Hq=20, Hkv=4, D=128, V=512, ctx=(800, 1500), model_nodes=(90, 120), n_chains=(1, 3),
         chain_len=8),
]


# "pair" copies Q tiles with TMA where the group divides 128; "pair-threads"
# forces the thread-written Q tiles (RS_DEBUG_ATTN_QCOPY=threads) everywhere
@pytest.mark.parametrize("form", ["pair", "pair-threads", "one"])
@pytest.mark.parametrize("kw", SHAPES, ids=[str(i) for i in range(len(SHAPES))])
def test_forms_every_row(kw, form, monkeypatch):
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", form.split("-")[0])
    if form == "pair-threads":
        monkeypatch.setenv("RS_DEBUG_ATTN_QCOPY", "threads")
    kw = dict(kw)
    seed = kw.pop("seed")
    w = synth.build(synth.small_spec(**kw), seed=seed)
    check_attn(w, make_step(w), rows=None)


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_pair_form_named(name, monkeypatch):
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    w = synth.make(name)
    check_attn(w, make_step(w), rows=None)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["gqa16k", "batched", "13b32k"])
def test_full_size_forms_agree(name, monkeypatch):
    # the default form is checked against the oracle on every row by
    # test_gpu_parity; here the other form must give the same outputs
    # within the oracle tolerance of each other
    w = synth.make(name)
    outs = {}
    for form in ("one", "pair"):
        monkeypatch.setenv("RS_DEBUG_ATTN_FORM", form)
        st = make_step(w)
        st.attn()
        torch.cuda.synchronize()
        assert (host(st.out["attn_status"]) == 0).all()
        outs[form] = (host(st.out["attn_out"]).astype(np.float64), host(st.out["attn_lse"]).astype(np.float64))
    (o1, l1), (o2, l2) = outs["one"], outs["pair"]
    assert np.abs(o1 - o2).max() <= 1e-2
    assert np.linalg.norm(o1 - o2) / np.linalg.norm(o1) <= 1e-2
    assert (np.abs(l1 - l2) / np.maximum(np.abs(l1), 1.0)).max() <= 1e-4


def test_pair_form_rejected_and_straddling_trees(monkeypatch):
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    rng = np.random.default_rng(5)
    Hq, Hkv, D = 16, 2, 128
    trees = [[-1, 0, 0, 1, 3], [-1, 0, 2, 1], [], [-1] + [int(rng.integers(0, i)) for i in range(1, 300)],
             [-1] + list(range(0, 99)), [-1] + [int(rng.integers(0, i)) for i in range(1, 70)]]
    S = [130, 50, 10, 200, 90, 1000]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert status.tolist() == [0, rs.RS_ST_BAD_TREE, 0, rs.RS_ST_TOO_LARGE, 0, 0]
    q, k, v, kv_off, ctx, node_off, parents = inp
    for b in (1, 3):
        n0, n1 = node_off[b], node_off[b + 1]
        assert (out[n0:n1] == 0).all() and (lse[n0:n1] == 0).all()
    for b in (0, 4, 5):
        n0, n1 = int(node_off[b]), int(node_off[b + 1])
        rows = [(n, h) for n in range(n0, n1) for h in range(Hq)]
        ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5, rows=rows)
        assert np.abs(out[n0:n1].reshape(-1, D) - ref["out"]).max() < 1e-2
        assert np.abs(lse[n0:n1].reshape(-1) - ref["lse"]).max() < 1e-3


def test_pair_form_many_requests(monkeypatch):
    # a few hundred requests of 1-40 nodes in groups of 8: many short
    # segments over the cost-weighted split, some CTA ranges empty
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    rng = np.random.default_rng(6)
    Hq, Hkv, D, B = 8, 1, 128, 300
    trees = []
    for _ in range(B):
        n = int(rng.integers(1, 41))
        trees.append([-1] + [int(rng.integers(0, i)) for i in range(1, n)])
    S = [int(x) for x in rng.integers(0, 400, B)]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert (status == 0).all()
    q, k, v, kv_off, ctx, node_off, parents = inp
    R = int(node_off[-1])
    rows = [(n, h) for n in range(R) for h in range(Hq)]
    ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5, rows=rows)
    assert np.abs(out.reshape(-1, D) - ref["out"]).max() < 1e-2


def test_pair_form_time_out_reports_status_and_recovers(monkeypatch):
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    rng = np.random.default_rng(7)
    Hq, Hkv, D = 16, 2, 128
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


def test_pair_form_empty_prefix_and_single_nodes(monkeypatch):
    # requests with no committed prefix (the first tile is all tree slots)
    # and single-node trees, in groups of 8 (half pairs and a full pair)
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    rng = np.random.default_rng(8)
    Hq, Hkv, D = 16, 2, 128
    trees = [[-1] + [int(rng.integers(0, i)) for i in range(1, 40)], [-1], [-1, 0, 1, 2], [-1],
             [-1] + [int(rng.integers(0, i)) for i in range(1, 20)]]
    S = [0, 0, 300, 1, 0]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert (status == 0).all()
    q, k, v, kv_off, ctx, node_off, parents = inp
    ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5)
    assert np.abs(out.reshape(-1, D) - ref["out"]).max() < 1e-2
    assert np.abs(lse.reshape(-1) - ref["lse"]).max() < 1e-3


def test_one_tile_form_streaming_launch_every_row(monkeypatch):
    # K/V larger than half the L2 makes the launch stream it (evict-first
    # copies, epilogue rows staged through shared memory): a small tree over
    # long prefixes, every (node, head) row against the oracle
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "one")
    kw = dict(B=2, Hq=8, Hkv=8, D=128, V=512, ctx=(20000, 22000), model_nodes=(20, 30), n_chains=(1, 2),
              chain_len=6)
    w = synth.build(synth.small_spec(**kw), seed=27)
    kv_bytes = 2 * w.k.shape[0] * 8 * 128 * 2
    l2 = getattr(torch.cuda.get_device_properties(0), "L2_cache_size", 129 * 2 ** 20)
    assert kv_bytes > 0.5 * l2
    check_attn(w, make_step(w), rows=None)


def test_pair_form_streaming_launch_every_row(monkeypatch):
    # K/V larger than half the L2 makes a pair-form launch stream it (evict-
    # first copies, the streaming split weights, every CTA's first Q copied
    # after its second K/V tile): GQA 4 over a few hundred tree nodes and long
    # prefixes, every (node, head) row against the oracle
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    kw = dict(B=2, Hq=32, Hkv=8, D=128, V=512, ctx=(20000, 21000), model_nodes=(90, 110), n_chains=(1, 2),
              chain_len=6)
    w = synth.build(synth.small_spec(**kw), seed=28)
    kv_bytes = 2 * w.k.shape[0] * 8 * 128 * 2
    l2 = getattr(torch.cuda.get_device_properties(0), "L2_cache_size", 129 * 2 ** 20)
    assert kv_bytes > 0.5 * l2
    assert int(np.diff(w.node_off).max()) * 4 > 128  # more than one row tile per KV head
    check_attn(w, make_step(w), rows=None)


@pytest.mark.parametrize("form", ["pair", "one"])
def test_row_counts_at_tile_edges(form, monkeypatch):
    # (node, head-in-group) rows per KV head of exactly one tile, one tile and
    # one node, exactly two tiles and two tiles and one node (G = 8: 16, 17,
    # 32 and 33 nodes): half pairs, full pairs with a short second tile and
    # pairs followed by a half pair, with prefixes that end on, just before
    # and just after a 128-key boundary
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", form)
    rng = np.random.default_rng(9)
    Hq, Hkv, D = 16, 2, 128
    trees = []
    for n in (16, 17, 32, 33):
        trees.append([-1] + [int(rng.integers(max(0, i - 3), i)) for i in range(1, n)])
    S = [256, 255, 257, 640]
    inp = _attn_inputs(rng, Hq, Hkv, D, S, trees)
    out, lse, status = _run_attn(*inp, Hq, Hkv, D, D ** -0.5)
    assert (status == 0).all()
    q, k, v, kv_off, ctx, node_off, parents = inp
    ref = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, D ** -0.5)
    assert np.abs(out.reshape(-1, D) - ref["out"]).max() < 1e-2
    assert np.linalg.norm(out.reshape(-1, D) - ref["out"]) / np.linalg.norm(ref["out"]) < 1e-2
    assert np.abs(lse.reshape(-1) - ref["lse"]).max() < 1e-3
