"""Seeded synthetic inputs shaped like the paper's workloads.

The paper measures on Spec-Bench with Vicuna-7B, Llama-3.1-8B and Qwen2-7B
(Section 4.1).  Neither the data nor the weights are available, so every
input here is drawn from a seeded PCG64 generator with the shapes, sizes and
structure of those runs; nothing from the benchmark itself is reproduced.

Recipe (per request b, generator PCG64(seed * 1000 + b)):

* token buffer of t = S + 1 tokens (the committed context plus the root token,
  i.e. the last committed token, whose KV is the first tree slot).  Ids are
  uniform in [0, V) and a config-specific share of the buffer is copied from
  earlier in the same buffer (planted repeats).  The last ``l`` tokens (the
  longest possible retrieval key) are additionally planted in front of each
  retrieved chain's origin, so every key length finds matches;
* draft tree, nodes in topological order: root, the model-draft tree level by
  level (given widths; node j of a level hangs from node floor(w_prev *
  (j / w)^2) of the previous level, so early branches are bushier), then each
  retrieved chain as a path from the root whose tokens are the buffer's
  continuation after the chain's origin;
* logits [N, V] fp32: standard normals times a per-row inverse temperature
  (log-uniform between sqrt(2 (ln V - 8)) and 40, which spreads the row
  entropies over roughly 0.1-8 nats), or N(0, 2^2) for the tiny case; then,
  per parent row, each child token is drawn "greedy" (prob 0.6, at most one
  per row: its logit is set to the row max + U(0.1, 1)), "close" (prob 0.2:
  row max - U(0, tau)) or left alone; optionally a tie at the row maximum is
  injected at another id;
* Q [N, Hq, D], K and V [S + N, Hkv, D]: N(0, 1) rounded to bf16 (K and V
  in 2048-row chunks, each from its own PCG64 stream seeded by (seed,
  request, tensor, chunk), generated in parallel);
* score table parallel to the buffer: 0.5 (the paper's S0), with a share of
  positions redrawn uniform in [0, 1] so the threshold filter and the ranking
  both have work to do;
* entropy history: l values uniform in [0.05, 3] nats; the previous step's
  committed rows are the root and the path to a random model node.

Nothing here computes an entropy, a match, an attention output or an
acceptance decision.
"""
from __future__ import annotations

import concurrent.futures as cf
import dataclasses
import math
import os
from functools import lru_cache
from typing import Optional, Sequence

import numpy as np


# --------------------------------------------------------------------- bf16
def bf16_bits(x: np.ndarray, out: Optional[np.ndarray] = None) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = np.right_shift(u, 16)
    np.bitwise_and(r, 1, out=r)
    np.add(r, 0x7FFF, out=r)
    np.add(r, u, out=r)
    np.right_shift(r, 16, out=r)
    if out is None:
        return r.astype(np.uint16)
    np.copyto(out, r.reshape(out.shape), casting="unsafe")
    return out


def bf16_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# --------------------------------------------------------------------- specs
@dataclasses.dataclass(frozen=True)
class Spec:
    name: str
    B: int
    Hq: int
    Hkv: int
    D: int
    V: int
    ctx: tuple                       # (lo, hi) context length S_b, inclusive
    model_widths: Optional[tuple]    # widths per depth; None = random (see model_nodes)
    model_nodes: tuple = (0, 0)      # (lo, hi) total tree nodes minus root, when random
    max_depth: int = 6
    n_chains: tuple = (1, 1)         # (lo, hi) retrieved chains per request
    chain_len: int = 8
    top_c: int = 3
    l: int = 3
    repeat_prob: float = 0.2         # share of buffer segments copied from earlier
    seg_len: tuple = (8, 64)         # (lo, hi) segment length
    logit_rule: str = "entropy"      # "entropy" or "gauss2"
    ties: bool = False
    score_noise: float = 0.3
    pos_cap: int = 1024
    # method hyper-parameters (Section 3; defaults where the paper gives none)
    lambda_e: float = 0.5
    theta_entropy: float = 1.5
    alpha: float = 0.3
    theta_score: float = 0.3
    beta: int = 5
    tau: float = 3.0
    phi: int = 2
    m: int = 2

    def params(self) -> dict:
        return dict(l=self.l, lambda_e=self.lambda_e, theta_entropy=self.theta_entropy,
                    alpha=self.alpha, theta_score=self.theta_score, top_c=self.top_c,
                    span_len=self.chain_len, beta=self.beta, tau=self.tau, phi=self.phi,
                    m=self.m)


CONFIGS = {
    # 1 layer, 4/4 heads x 64, context 256, root + model chain 4 + retrieved chain 4
    "tiny": Spec("tiny", B=1, Hq=4, Hkv=4, D=64, V=1024, ctx=(256, 256),
                 model_widths=(1, 1, 1, 1), n_chains=(1, 1), chain_len=4, top_c=3, l=3,
                 repeat_prob=0.0, logit_rule="gauss2", ties=True, score_noise=0.0),
    # 32/32 x 128, context 2048, 16-node model tree + 3 chains of 8, V=32000
    "7b": Spec("7b", B=1, Hq=32, Hkv=32, D=128, V=32000, ctx=(2048, 2048),
               model_widths=(4, 4, 3, 3, 2), n_chains=(3, 3), chain_len=8, top_c=3, l=3,
               repeat_prob=0.2, seg_len=(8, 64)),
    # 32/8 x 128, context 16384, 16-node model tree + 8 chains of 16, V=128256
    "gqa16k": Spec("gqa16k", B=1, Hq=32, Hkv=8, D=128, V=128256, ctx=(16384, 16384),
                   model_widths=(4, 4, 3, 3, 2), n_chains=(8, 8), chain_len=16, top_c=8, l=3,
                   repeat_prob=0.5, seg_len=(64, 64)),
    # 16 requests, 32/8 x 128, contexts U[1024, 8192], 24-64 draft nodes, V=128256, l=4
    "batched": Spec("batched", B=16, Hq=32, Hkv=8, D=128, V=128256, ctx=(1024, 8192),
                    model_widths=None, model_nodes=(24, 64), max_depth=6, n_chains=(0, 3),
                    chain_len=8, top_c=3, l=4, repeat_prob=0.2, seg_len=(8, 64)),
    # 4 requests, 40/40 x 128, context 32768, 32-node model tree + 4 chains of 8, V=32000
    "13b32k": Spec("13b32k", B=4, Hq=40, Hkv=40, D=128, V=32000, ctx=(32768, 32768),
                   model_widths=(8, 8, 6, 5, 5), n_chains=(4, 4), chain_len=8, top_c=4, l=3,
                   repeat_prob=0.3, seg_len=(8, 64)),
}


def small_spec(name="small", **kw) -> Spec:
    """A parity-test sized spec; keyword arguments override the defaults."""
    base = dict(name=name, B=3, Hq=8, Hkv=2, D=128, V=3000, ctx=(100, 700),
                model_widths=None, model_nodes=(5, 40), max_depth=5, n_chains=(0, 3),
                chain_len=6, top_c=3, l=3, repeat_prob=0.3, seg_len=(4, 24), ties=True)
    base.update(kw)
    return Spec(**base)


# --------------------------------------------------------------------- workload
@dataclasses.dataclass
class Workload:
    spec: Spec
    seed: int
    # token buffers and scores (parallel), offsets [B+1]
    tokens: np.ndarray
    tok_off: np.ndarray
    scores: np.ndarray
    # tree, node offsets [B+1]
    node_off: np.ndarray
    parents: np.ndarray
    tree_tokens: np.ndarray
    source: np.ndarray
    chain: np.ndarray
    sel_pos: np.ndarray        # [B, top_c] chain origins (-1 = none)
    # attention
    q: np.ndarray              # [R, Hq, D] bf16 bits
    k: np.ndarray              # [T, Hkv, D] bf16 bits
    v: np.ndarray
    kv_off: np.ndarray         # [B] int64
    ctx_len: np.ndarray        # [B] int32
    # logits and gate state
    logits: np.ndarray         # [R, V] f32
    row_commit: np.ndarray     # [R] u8
    hist: np.ndarray           # [B, l] f32
    hist_n: np.ndarray         # [B] i32
    k_star_hint: np.ndarray    # [B] i32 key lengths for stand-alone scans

    @property
    def B(self):
        return self.spec.B

    @property
    def R(self):
        return int(self.node_off[-1])

    def params(self):
        return self.spec.params()


_KV_CHUNK_ROWS = 2048


def _fill_normal_bf16(dst: np.ndarray, key: tuple):
    """dst[...] = N(0, 1) rounded to bf16, in row chunks generated in parallel;
    chunk j uses PCG64(SeedSequence(key + (j,))), so the values do not depend
    on the number of threads."""
    rows = dst.shape[0]
    chunks = list(range(0, rows, _KV_CHUNK_ROWS))

    def work(j0):
        n = min(_KV_CHUNK_ROWS, rows - j0)
        g = np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(key) + [j0])))
        x = g.standard_normal((n,) + dst.shape[1:], dtype=np.float32)
        bf16_bits(x, out=dst[j0:j0 + n])

    if len(chunks) <= 2:
        for j0 in chunks:
            work(j0)
        return
    with cf.ThreadPoolExecutor(max_workers=min(len(chunks), os.cpu_count() or 4)) as ex:
        list(ex.map(work, chunks))


def _model_widths(rng, spec: Spec, n_model: int):
    if spec.model_widths is not None:
        return list(spec.model_widths)
    if n_model <= 0:
        return []
    depth = min(spec.max_depth, n_model)
    w = [1] * depth
    extra = n_model - depth
    if extra > 0:
        pref = np.array([1.0 / (d + 1) for d in range(depth)])
        w = list(np.array(w) + rng.multinomial(extra, pref / pref.sum()))
    return [int(x) for x in w]


def _token_buffer(rng, spec: Spec, t: int, V: int):
    X = rng.integers(0, V, size=t, dtype=np.int64).astype(np.int32)
    if spec.name == "tiny" or spec.repeat_prob <= 0:
        # 3 planted 6-token spans, each copied to a second place; the buffer
        # tail is set to a planted span's prefix
        spans = []
        for s in range(3):
            src = 10 + s * 60
            dst = src + 30
            X[dst:dst + 6] = X[src:src + 6]
            spans.append(src)
        X[t - 3:t] = X[spans[0]:spans[0] + 3]
        return X
    p = 0
    lo, hi = spec.seg_len
    while p < t:
        n = int(rng.integers(lo, hi + 1))
        n = min(n, t - p)
        if p > n and rng.random() < spec.repeat_prob:
            src = int(rng.integers(0, p - n + 1))
            X[p:p + n] = X[src:src + n]
        p += n
    return X


def _plant_row(rng, z, child_tokens, tau, ties):
    """Per parent row: at most one greedy child, some close children."""
    zmax = float(z.max())
    labels = rng.random(len(child_tokens))
    greedy_done = False
    close = []
    for tok, u in zip(child_tokens, labels):
        if u < 0.6 and not greedy_done:
            z[tok] = np.float32(zmax + rng.uniform(0.1, 1.0))
            greedy_done = True
        elif u < 0.8 or (u < 0.6 and greedy_done):
            close.append(tok)
    top = float(z.max())
    for tok in close:
        z[tok] = np.float32(top - rng.uniform(0.0, tau))
    if ties and rng.random() < 0.25:
        other = int(rng.integers(0, z.size))
        z[other] = z.max()


def _request(spec: Spec, rng, S: int):
    l, L = spec.l, spec.chain_len
    t = S + 1
    X = _token_buffer(rng, spec, t, spec.V)

    # draft tree sizes
    if spec.model_widths is not None:
        nch = int(rng.integers(spec.n_chains[0], spec.n_chains[1] + 1))
        widths = _model_widths(rng, spec, sum(spec.model_widths))
    else:
        n_draft = int(rng.integers(spec.model_nodes[0], spec.model_nodes[1] + 1))
        nch = int(rng.integers(spec.n_chains[0], spec.n_chains[1] + 1))
        nch = min(nch, n_draft // L, spec.top_c)
        widths = _model_widths(rng, spec, n_draft - nch * L)
    nch = min(nch, spec.top_c)

    # chain origins: the key (last l tokens) is planted in front of each
    origins = []
    lo_p, hi_p = l + 1, t - 2 - L - l - 1
    if hi_p > lo_p:
        for _ in range(200):
            if len(origins) == nch:
                break
            p = int(rng.integers(lo_p, hi_p))
            if all(abs(p - o) > L + l + 1 for o in origins):
                origins.append(p)
    key = X[t - l:t].copy()
    for p in origins:
        X[p - l + 1:p + 1] = key
    nch = len(origins)

    # tree: root, model levels, chains
    parents = [-1]
    source = [0]
    chain = [-1]
    toks = [int(X[t - 1])]
    prev = [0]
    for w in widths:
        cur = []
        wp = len(prev)
        sib_used = {}
        for j in range(w):
            pi = prev[min(wp - 1, int(math.floor(wp * (j / w) ** 2)))]
            used = sib_used.setdefault(pi, set())
            tok = int(rng.integers(0, spec.V))
            while tok in used:
                tok = int(rng.integers(0, spec.V))
            used.add(tok)
            parents.append(pi)
            source.append(1)
            chain.append(-1)
            toks.append(tok)
            cur.append(len(parents) - 1)
        prev = cur
    sel = [-1] * spec.top_c
    for c, p in enumerate(origins):
        n_tok = min(L, t - 1 - p)
        par = 0
        for j in range(n_tok):
            parents.append(par)
            source.append(2)
            chain.append(c)
            toks.append(int(X[p + 1 + j]))
            par = len(parents) - 1
        sel[c] = p
    N = len(parents)
    return dict(X=X, t=t, S=S, N=N, parents=np.array(parents, np.int32),
                source=np.array(source, np.uint8), chain=np.array(chain, np.int8),
                toks=np.array(toks, np.int32), sel=np.array(sel, np.int32), widths=widths)


def build(spec: Spec, seed: int = 0) -> Workload:
    reqs = []
    for b in range(spec.B):
        rng = np.random.Generator(np.random.PCG64(seed * 1000 + b))
        S = int(rng.integers(spec.ctx[0], spec.ctx[1] + 1))
        r = _request(spec, rng, S)
        r["rng"] = rng
        reqs.append(r)

    B = spec.B
    tok_off = np.zeros(B + 1, np.int64)
    node_off = np.zeros(B + 1, np.int32)
    kv_off = np.zeros(B, np.int64)
    for b, r in enumerate(reqs):
        tok_off[b + 1] = tok_off[b] + r["t"]
        node_off[b + 1] = node_off[b] + r["N"]
        if b + 1 < B:
            kv_off[b + 1] = kv_off[b] + r["S"] + r["N"]
    T = int(kv_off[-1] + reqs[-1]["S"] + reqs[-1]["N"]) if B else 0
    R = int(node_off[-1])

    tokens = np.concatenate([r["X"] for r in reqs]).astype(np.int32)
    parents = np.concatenate([r["parents"] for r in reqs])
    source = np.concatenate([r["source"] for r in reqs])
    chain = np.concatenate([r["chain"] for r in reqs])
    tree_tokens = np.concatenate([r["toks"] for r in reqs])
    sel_pos = np.stack([r["sel"] for r in reqs]).astype(np.int32)
    ctx_len = np.array([r["S"] for r in reqs], np.int32)

    q = np.empty((R, spec.Hq, spec.D), np.uint16)
    k = np.empty((T, spec.Hkv, spec.D), np.uint16)
    v = np.empty((T, spec.Hkv, spec.D), np.uint16)
    logits = np.empty((R, spec.V), np.float32)
    scores = np.full(int(tok_off[-1]), 0.5, np.float32)
    row_commit = np.zeros(R, np.uint8)
    hist = np.zeros((B, spec.l), np.float32)
    hist_n = np.zeros(B, np.int32)
    k_hint = np.zeros(B, np.int32)

    for b, r in enumerate(reqs):
        rng = r["rng"]
        n0, N, S = int(node_off[b]), r["N"], r["S"]
        q[n0:n0 + N] = bf16_bits(rng.standard_normal((N, spec.Hq, spec.D), dtype=np.float32))
        _fill_normal_bf16(k[int(kv_off[b]):int(kv_off[b]) + S + N], (seed, b, 0))
        _fill_normal_bf16(v[int(kv_off[b]):int(kv_off[b]) + S + N], (seed, b, 1))

        # logits with planted acceptance structure
        z = rng.standard_normal((N, spec.V), dtype=np.float32)
        if spec.logit_rule == "gauss2":
            z *= np.float32(2.0)
        else:
            blo = math.sqrt(max(2.0 * (math.log(spec.V) - 8.0), 0.25))
            beta_r = np.exp(rng.uniform(math.log(blo), math.log(40.0), size=N)).astype(np.float32)
            z *= beta_r[:, None]
        par = r["parents"]
        children = {}
        for i in range(1, N):
            children.setdefault(int(par[i]), []).append(int(r["toks"][i]))
        for p_row in range(N):
            ch = children.get(p_row, [])
            if ch:
                _plant_row(rng, z[p_row], ch, spec.tau, spec.ties)
            elif spec.ties and rng.random() < 0.1:
                z[p_row, int(rng.integers(0, spec.V))] = z[p_row].max()
        logits[n0:n0 + N] = z

        # scores: S0 plus a redrawn share
        t0, t = int(tok_off[b]), r["t"]
        if spec.score_noise > 0:
            mask = rng.random(t) < spec.score_noise
            scores[t0:t0 + t][mask] = rng.random(int(mask.sum())).astype(np.float32)

        # previous step's committed rows: root + path to a random model node
        row_commit[n0] = 1
        model_nodes = np.nonzero(r["source"] == 1)[0]
        if model_nodes.size:
            a = int(rng.choice(model_nodes))
            while a > 0:
                row_commit[n0 + a] = 1
                a = int(par[a])
        hist[b] = rng.uniform(0.05, 3.0, size=spec.l).astype(np.float32)
        hist_n[b] = spec.l if rng.random() < 0.8 else int(rng.integers(0, spec.l + 1))
        k_hint[b] = int(rng.integers(1, spec.l + 1))

    return Workload(spec=spec, seed=seed, tokens=tokens, tok_off=tok_off, scores=scores,
                    node_off=node_off, parents=parents, tree_tokens=tree_tokens, source=source,
                    chain=chain, sel_pos=sel_pos, q=q, k=k, v=v, kv_off=kv_off, ctx_len=ctx_len,
                    logits=logits, row_commit=row_commit, hist=hist, hist_n=hist_n,
                    k_star_hint=k_hint)


@lru_cache(maxsize=4)
def make(name: str, seed: int = 0) -> Workload:
    """One of the named configurations (cached per process)."""
    return build(CONFIGS[name], seed)
