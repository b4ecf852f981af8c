"""Pins for the oracle's tree-verification attention.

The oracle walks parent links per node; these tests build the tree mask a
different way (children lists, depth-first from the root) and compare with
PyTorch's scaled_dot_product_attention in fp64 on the CPU, and check the
special cases the definition fixes: a chain is causal attention, a single
node is plain decode attention, GQA equals MHA with repeated KV heads,
prefix order does not matter, and two hand-worked cases
(tests/golden/attn_cases.json).
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth


def _f64(bits):
    return torch.from_numpy(synth.bf16_to_f32(bits).astype(np.float64))


def _ancestor_mask(parents):
    """mask[i, a] = a is on the root-to-i path, via DFS over children lists."""
    N = len(parents)
    kids = [[] for _ in range(N)]
    for i in range(1, N):
        kids[parents[i]].append(i)
    mask = np.zeros((N, N), bool)
    stack = [(0, [0])]
    while stack:
        node, path = stack.pop()
        mask[node, path] = True
        for c in kids[node]:
            stack.append((c, path + [c]))
    return mask


def _sdpa_reference(w_q, w_k, w_v, kv_off, ctx_len, node_off, parents, Hq, Hkv, D, scale):
    """Per request and head, SDPA with an explicit boolean mask (fp64)."""
    G = Hq // Hkv
    R = int(node_off[-1])
    out = np.zeros((R, Hq, D))
    lse = np.zeros((R, Hq))
    for b in range(len(node_off) - 1):
        n0, n1 = int(node_off[b]), int(node_off[b + 1])
        N, S = n1 - n0, int(ctx_len[b])
        k0 = int(kv_off[b])
        mask = np.ones((N, S + N), bool)
        mask[:, S:] = _ancestor_mask(parents[n0:n1])
        m = torch.from_numpy(mask)
        for h in range(Hq):
            q = _f64(w_q[n0:n1, h])
            k = _f64(w_k[k0:k0 + S + N, h // G])
            v = _f64(w_v[k0:k0 + S + N, h // G])
            o = torch.nn.functional.scaled_dot_product_attention(
                q[None, None], k[None, None], v[None, None], attn_mask=m[None, None], scale=scale)
            out[n0:n1, h] = o[0, 0].numpy()
            s = (q @ k.T) * scale
            s = s.masked_fill(~m, -math.inf)
            lse[n0:n1, h] = torch.logsumexp(s, dim=-1).numpy()
    return out, lse


def _rand_case(seed, B, Hq, Hkv, D, S_list, trees):
    rng = np.random.default_rng(seed)
    node_off = np.concatenate([[0], np.cumsum([len(t) for t in trees])]).astype(np.int32)
    kv_off = np.concatenate([[0], np.cumsum([s + len(t) for s, t in zip(S_list, trees)])[:-1]])
    T = sum(s + len(t) for s, t in zip(S_list, trees))
    R = int(node_off[-1])
    q = synth.bf16_bits(rng.standard_normal((R, Hq, D)).astype(np.float32))
    k = synth.bf16_bits(rng.standard_normal((T, Hkv, D)).astype(np.float32))
    v = synth.bf16_bits(rng.standard_normal((T, Hkv, D)).astype(np.float32))
    parents = np.concatenate([np.array(t, np.int32) for t in trees])
    return q, k, v, kv_off.astype(np.int64), np.array(S_list, np.int32), node_off, parents


def _run(case, Hq, Hkv, D, scale):
    q, k, v, kv_off, ctx, node_off, parents = case
    o = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, parents, Hq, Hkv, D, scale)
    R = int(node_off[-1])
    assert o["rc"] == 0
    return o["out"].reshape(R, Hq, D), o["lse"].reshape(R, Hq)


def test_golden(golden_dir):
    for c in json.load(open(os.path.join(golden_dir, "attn_cases.json")))["cases"]:
        D, Hq, Hkv = c["D"], c["Hq"], c["Hkv"]
        q = synth.bf16_bits(np.array(c["q"], np.float32))
        k = synth.bf16_bits(np.array(c["k"], np.float32))
        v = synth.bf16_bits(np.array(c["v"], np.float32))
        N = len(c["parents"])
        out, lse = _run((q, k, v, np.array([0]), np.array([c["ctx_len"]]), np.array([0, N]),
                         np.array(c["parents"])), Hq, Hkv, D, c["scale"])
        np.testing.assert_allclose(out, np.array(c["out"]), rtol=1e-14, atol=1e-15, err_msg=c["name"])
        np.testing.assert_allclose(lse, np.array(c["lse"]), rtol=1e-14, atol=1e-15, err_msg=c["name"])


def test_chain_is_causal_attention():
    N, S, D = 7, 33, 64
    case = _rand_case(1, 1, 2, 2, D, [S], [[-1] + list(range(N - 1))])
    out, lse = _run(case, 2, 2, D, D ** -0.5)
    q, k, v = (_f64(a) for a in case[:3])
    for h in range(2):
        # causal over the sequence prefix + chain: query i sees keys < S + i + 1
        mask = torch.arange(S + N)[None, :] < (S + torch.arange(N)[:, None] + 1)
        ref = torch.nn.functional.scaled_dot_product_attention(
            q[None, None, :, h], k[None, None, :, h], v[None, None, :, h], attn_mask=mask[None, None],
            scale=D ** -0.5)[0, 0]
        np.testing.assert_allclose(out[:, h], ref.numpy(), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("seed", [2, 3])
def test_tree_matches_masked_sdpa(seed):
    rng = np.random.default_rng(seed)
    trees = []
    for n in (1, 12, 30):
        trees.append([-1] + [int(rng.integers(0, i)) for i in range(1, n)])
    S_list = [0, 17, 130]
    Hq, Hkv, D = 6, 3, 64
    case = _rand_case(seed, 3, Hq, Hkv, D, S_list, trees)
    out, lse = _run(case, Hq, Hkv, D, 0.125)
    ref_o, ref_l = _sdpa_reference(*case, Hq, Hkv, D, 0.125)
    np.testing.assert_allclose(out, ref_o, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(lse, ref_l, rtol=1e-12, atol=1e-12)


def test_tree_equals_per_branch_decode():
    # each root-to-leaf path, laid out as its own chain request, gives the
    # same outputs for every node on it
    parents = [-1, 0, 0, 1, 1, 2, 4, 4]
    S, Hq, D = 20, 2, 64
    case = _rand_case(4, 1, Hq, Hq, D, [S], [parents])
    out, _ = _run(case, Hq, Hq, D, 0.1)
    q, k, v = case[:3]
    leaves = [i for i in range(len(parents)) if i not in parents]
    for leaf in leaves:
        path = []
        a = leaf
        while a != -1:
            path.append(a)
            a = parents[a]
        path = path[::-1]
        kk = np.concatenate([k[:S], k[S + np.array(path)]])
        vv = np.concatenate([v[:S], v[S + np.array(path)]])
        sub = (q[path], kk, vv, np.array([0]), np.array([S], np.int32),
               np.array([0, len(path)], np.int32), np.array([-1] + list(range(len(path) - 1)), np.int32))
        o2, _ = _run(sub, Hq, Hq, D, 0.1)
        np.testing.assert_allclose(o2, out[path], rtol=1e-13, atol=1e-14)


def test_single_node_is_decode_attention():
    S, D = 50, 128
    case = _rand_case(5, 1, 4, 1, D, [S], [[-1]])
    out, lse = _run(case, 4, 1, D, D ** -0.5)
    q, k, v = (_f64(a) for a in case[:3])
    for h in range(4):
        ref = torch.nn.functional.scaled_dot_product_attention(
            q[None, None, :, h], k[None, None, :, 0], v[None, None, :, 0], scale=D ** -0.5)[0, 0]
        np.testing.assert_allclose(out[:, h], ref.numpy(), rtol=1e-12, atol=1e-13)
        s = (q[:, h] @ k[:, 0].T) * D ** -0.5
        np.testing.assert_allclose(lse[:, h], torch.logsumexp(s, -1).numpy(), rtol=1e-13)


def test_gqa_equals_mha_with_repeated_kv():
    trees = [[-1, 0, 1, 0, 3]]
    Hq, Hkv, D = 8, 2, 64
    q, k, v, kv_off, ctx, node_off, parents = _rand_case(6, 1, Hq, Hkv, D, [40], trees)
    out, lse = _run((q, k, v, kv_off, ctx, node_off, parents), Hq, Hkv, D, 0.2)
    kr = np.repeat(k, Hq // Hkv, axis=1)
    vr = np.repeat(v, Hq // Hkv, axis=1)
    out2, lse2 = _run((q, kr, vr, kv_off, ctx, node_off, parents), Hq, Hq, D, 0.2)
    np.testing.assert_allclose(out, out2, rtol=0, atol=0)
    np.testing.assert_allclose(lse, lse2, rtol=0, atol=0)


def test_prefix_permutation_invariance():
    trees = [[-1, 0, 0, 2]]
    S, D = 60, 64
    q, k, v, kv_off, ctx, node_off, parents = _rand_case(7, 1, 2, 2, D, [S], trees)
    out, lse = _run((q, k, v, kv_off, ctx, node_off, parents), 2, 2, D, 0.125)
    perm = np.random.default_rng(0).permutation(S)
    k2 = k.copy()
    v2 = v.copy()
    k2[:S] = k[perm]
    v2[:S] = v[perm]
    out2, lse2 = _run((q, k2, v2, kv_off, ctx, node_off, parents), 2, 2, D, 0.125)
    np.testing.assert_allclose(out, out2, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(lse, lse2, rtol=1e-14)


def test_tiny_workload_matches_sdpa():
    w = synth.make("tiny")
    s = w.spec
    o = oracle.tree_attn(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents,
                         s.Hq, s.Hkv, s.D, s.D ** -0.5)
    ref_o, ref_l = _sdpa_reference(w.q, w.k, w.v, w.kv_off, w.ctx_len, w.node_off, w.parents,
                                   s.Hq, s.Hkv, s.D, s.D ** -0.5)
    np.testing.assert_allclose(o["out"].reshape(ref_o.shape), ref_o, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(o["lse"].reshape(ref_l.shape), ref_l, rtol=1e-12)


def test_malformed_parents_are_reported():
    q, k, v, kv_off, ctx, node_off, _ = _rand_case(8, 1, 1, 1, 64, [4], [[-1, 0, 1]])
    o = oracle.tree_attn(q, k, v, kv_off, ctx, node_off, np.array([-1, 2, 1], np.int32), 1, 1, 64, 0.1)
    assert o["rc"] == 1
