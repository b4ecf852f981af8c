"""Synthetic end-to-end loop of Algorithm 1 over many decoding steps.

A random-weight decoder-only transformer (GQA, head dim 64, no positional
encoding, RMSNorm, SwiGLU MLP, an untied output head scaled to logits of
standard deviation ~6, which gives rows a median entropy of ~1.8 nats) plays
the target model; the
same architecture with perturbed weights plays the draft model.  Both run
their attention through ``rs_tree_verify_attn`` over a bf16 KV cache (the
committed prefix, then the draft tree's slots); projections and MLPs are
plain torch matmuls.  Every step:

  1. trigger: ``rs_entropy_gate_rows`` on the previous verify's row entropies
     (k*, entropy_ok; nothing fires until the history has entries);
  2. retrieval: ``rs_match_scan`` over the committed tokens (or, with
     ``retrieval="index"``, ``rs_match_scan_indexed`` on an index that
     ``rs_match_index_append`` brings up to date) -> up to top_c
     continuations, attached under the root as retrieved chains;
  3. model drafts: the draft model expands a top-w tree level by level;
  4. verification: one target forward over the whole tree, then
     ``rs_accept`` (strict for model drafts, relaxed + look-ahead for chains,
     EMA of the selected positions' scores, row entropies);
  5. commit: the accepted tokens and the bonus token are appended; the
     accepted slots' K/V are moved into the prefix.

With tau = 0 the relaxed check accepts only argmax tokens, so the loop must
reproduce the target's plain greedy decoding token for token
(``greedy_reference`` computes that with dense attention in torch).

``python -m paper_2511_01282_gb300.e2e --sweep`` prints the mean accepted
tokens per step, the trigger rate and the number of non-greedy tokens for a
grid of tau and m (the shape of the paper's sensitivity study, on synthetic
data and random weights).
"""
import argparse
import json
import math

import numpy as np
import torch

from . import respec as rs


def _rms(x, eps=1e-6):
    return x * torch.rsqrt(x.pow(2).mean(-1, keepdim=True) + eps)


class TinyLM:
    """Random-weight GQA decoder; attention through rs_tree_verify_attn."""

    def __init__(self, V=4096, d=256, L=2, Hq=4, Hkv=2, D=64, ffn=512, seed=0, logit_std=6.0,
                 base=None, noise=0.0, device="cuda"):
        self.V, self.d, self.L, self.Hq, self.Hkv, self.D = V, d, L, Hq, Hkv, D
        self.logit_scale = logit_std / math.sqrt(d)  # unit-RMS state, unit-variance head
        self.device = torch.device(device)
        g = torch.Generator().manual_seed(seed)

        def w(*shape):
            return torch.randn(*shape, generator=g) / math.sqrt(shape[0])

        names = ["emb", "head"] + ["%s.%d" % (n, i) for i in range(L)
                                   for n in ("wq", "wk", "wv", "wo", "w1", "w3", "w2")]
        shapes = {"emb": (V, d), "head": (d, V), "wq": (d, Hq * D), "wk": (d, Hkv * D), "wv": (d, Hkv * D),
                  "wo": (Hq * D, d), "w1": (d, ffn), "w3": (d, ffn), "w2": (ffn, d)}
        self.p = {}
        for n in names:
            key = n.split(".")[0]
            t = w(*shapes[key]) if key not in ("emb", "head") else torch.randn(*shapes[key], generator=g)
            if base is not None:
                t = base.p[n].cpu() + noise * torch.randn(t.shape, generator=g) * t.std()
            self.p[n] = t.to(self.device)

    # ------------------------------------------------------------ KV cache
    def new_cache(self, cap):
        z = lambda: torch.zeros((cap, self.Hkv, self.D), dtype=torch.bfloat16, device=self.device)  # noqa: E731
        return dict(K=[z() for _ in range(self.L)], V=[z() for _ in range(self.L)], cap=cap, S=0)

    def forward_tree(self, cache, tokens, parents, ws):
        """Logits [N, V] of a draft tree hanging after the cached prefix.

        tokens [N] int64, parents [N] int32 (local, -1 at the root), both on
        the device.  The tree's K/V are written to slots S .. S + N - 1."""
        N, S = tokens.numel(), cache["S"]
        assert S + N <= cache["cap"] and N <= 256
        dev = self.device
        kv_off = torch.zeros(1, dtype=torch.int64, device=dev)
        ctx = torch.full((1,), S, dtype=torch.int32, device=dev)
        node_off = torch.tensor([0, N], dtype=torch.int32, device=dev)
        out = torch.empty((N, self.Hq, self.D), dtype=torch.float32, device=dev)
        lse = torch.empty((N, self.Hq), dtype=torch.float32, device=dev)
        status = torch.empty(1, dtype=torch.int32, device=dev)
        x = self.p["emb"][tokens]
        for i in range(self.L):
            h = _rms(x)
            q = (h @ self.p["wq.%d" % i]).view(N, self.Hq, self.D).to(torch.bfloat16).contiguous()
            cache["K"][i][S:S + N] = (h @ self.p["wk.%d" % i]).view(N, self.Hkv, self.D).to(torch.bfloat16)
            cache["V"][i][S:S + N] = (h @ self.p["wv.%d" % i]).view(N, self.Hkv, self.D).to(torch.bfloat16)
            rs.rs_tree_verify_attn(q, cache["K"][i], cache["V"][i], cache["cap"], kv_off, ctx, node_off,
                                   parents, 1, N, self.Hq, self.Hkv, self.D, self.D ** -0.5, out, lse,
                                   status, ws)
            x = x + out.view(N, self.Hq * self.D) @ self.p["wo.%d" % i]
            h = _rms(x)
            x = x + (torch.nn.functional.silu(h @ self.p["w1.%d" % i]) * (h @ self.p["w3.%d" % i])) @ self.p["w2.%d" % i]
        return (_rms(x) @ self.p["head"]) * self.logit_scale

    def commit(self, cache, slots):
        """Move tree slots S + slots[j] to S + j (j in order) and grow the prefix."""
        S, n = cache["S"], len(slots)
        if n:
            src = torch.tensor([S + s for s in slots], dtype=torch.int64, device=self.device)
            for i in range(self.L):
                cache["K"][i][S:S + n] = cache["K"][i][src]
                cache["V"][i][S:S + n] = cache["V"][i][src]
        cache["S"] = S + n

    def dense_logits(self, tokens):
        """Plain causal attention over a whole sequence (bf16-rounded Q, K, V
        as in the cache, fp32 softmax): the independent greedy reference."""
        T = tokens.numel()
        x = self.p["emb"][tokens]
        G = self.Hq // self.Hkv
        mask = torch.ones((T, T), dtype=torch.bool, device=self.device).tril()
        for i in range(self.L):
            h = _rms(x)
            q = (h @ self.p["wq.%d" % i]).view(T, self.Hq, self.D).to(torch.bfloat16).float()
            k = (h @ self.p["wk.%d" % i]).view(T, self.Hkv, self.D).to(torch.bfloat16).float()
            v = (h @ self.p["wv.%d" % i]).view(T, self.Hkv, self.D).to(torch.bfloat16).float()
            k, v = k.repeat_interleave(G, dim=1), v.repeat_interleave(G, dim=1)
            s = torch.einsum("qhd,khd->hqk", q, k) * self.D ** -0.5
            s = s.masked_fill(~mask, float("-inf"))
            o = torch.einsum("hqk,khd->qhd", torch.softmax(s, -1), v)
            x = x + o.reshape(T, self.Hq * self.D) @ self.p["wo.%d" % i]
            h = _rms(x)
            x = x + (torch.nn.functional.silu(h @ self.p["w1.%d" % i]) * (h @ self.p["w3.%d" % i])) @ self.p["w2.%d" % i]
        return (_rms(x) @ self.p["head"]) * self.logit_scale


def greedy_reference(model, prompt, n_new):
    """Plain greedy decoding with dense attention (one token at a time)."""
    seq = torch.as_tensor(np.asarray(prompt), dtype=torch.int64, device=model.device)
    for _ in range(n_new):
        nxt = model.dense_logits(seq)[-1].argmax()
        seq = torch.cat([seq, nxt.view(1)])
    return seq.cpu().numpy()[len(prompt):]


class SpecLoop:
    """One request decoded by the full step of Algorithm 1 (B = 1)."""

    def __init__(self, target, draft, prompt, p, widths=(4, 3, 2), cap=4096, acc_cap=64, trace=False,
                 retrieval="scan"):
        self.t, self.dr, self.p = target, draft, p
        # retrieval: "scan" (rs_match_scan over the buffer) or "index" (an
        # index built over the prompt, the committed tokens appended to it
        # every step, queried with rs_match_scan_indexed)
        assert retrieval in ("scan", "index")
        self.retrieval = retrieval
        # with trace, every step appends host copies of each call's inputs and
        # outputs to self.trace (for checking a run call by call)
        self.trace = [] if trace else None
        self.widths = widths
        self.acc_cap = acc_cap
        dev = self.dev = target.device
        self.cap = cap
        prompt = np.asarray(prompt, np.int32)
        self.buf = torch.zeros(cap, dtype=torch.int32, device=dev)
        self.buf[:len(prompt)] = torch.from_numpy(prompt).to(dev)
        self.n = len(prompt)                       # committed tokens (the last is the root)
        self.scores = torch.full((cap,), 0.5, dtype=torch.float32, device=dev)
        self.hist = torch.zeros((1, p.l), dtype=torch.float32, device=dev)
        self.hist_n = torch.zeros(1, dtype=torch.int32, device=dev)
        self.k_star = torch.zeros(1, dtype=torch.int32, device=dev)
        self.h_best = torch.zeros(1, dtype=torch.float32, device=dev)
        self.ok = torch.zeros(1, dtype=torch.uint8, device=dev)
        self.tc = target.new_cache(cap)
        self.dc = draft.new_cache(cap)
        self.ws_attn = torch.empty(max(rs.rs_tree_verify_attn_workspace_size(1, 256, target.Hq, target.Hkv,
                                                                              target.D), 256),
                                   dtype=torch.uint8, device=dev)
        # prefill both caches with every prompt token but the root (chains of <= 256)
        for m in (target, draft):
            cache = self.tc if m is target else self.dc
            for a in range(0, len(prompt) - 1, 256):
                toks = self.buf[a:min(a + 256, len(prompt) - 1)].long()
                m.forward_tree(cache, toks, self._chain_parents(toks.numel()), self.ws_attn)
                m.commit(cache, list(range(toks.numel())))
        self.stats = dict(steps=0, emitted=0, triggered=0, retrieval_wins=0, model_wins=0, relaxed=0)
        if retrieval == "index":
            self.idx_t = len(prompt)
            self.idx = torch.empty(rs.rs_match_index_bytes(1, target.V, self.idx_t), dtype=torch.uint8, device=dev)
            self.idx_status = torch.zeros(1, dtype=torch.int32, device=dev)
            rs.rs_match_index_build(self.buf, torch.tensor([0, self.n], dtype=torch.int64, device=dev), 1, target.V,
                                    self.idx_t, self.idx)

    def _chain_parents(self, n):
        return torch.arange(-1, n - 1, dtype=torch.int32, device=self.dev)

    def _draft_tree(self, root):
        """Model drafts: top-w expansion level by level with the draft model."""
        toks, par = [root], [-1]
        frontier = [0]
        for w in self.widths:
            if not frontier or len(toks) + len(frontier) * w > 200:
                break
            logits = self.dr.forward_tree(self.dc, torch.tensor(toks, dtype=torch.int64, device=self.dev),
                                          torch.tensor(par, dtype=torch.int32, device=self.dev), self.ws_attn)
            top = logits[frontier].topk(w, dim=-1).indices.cpu().numpy()
            nxt = []
            for f, row in zip(frontier, top):
                for tok in row:
                    toks.append(int(tok))
                    par.append(f)
                    nxt.append(len(toks) - 1)
            frontier = nxt
        return toks, par

    def step(self):
        p, dev = self.p, self.dev
        tok_off = torch.tensor([0, self.n], dtype=torch.int64, device=dev)
        root = int(self.buf[self.n - 1])
        # 2. retrieval, gated by the trigger of the previous step
        top_c, L = p.top_c, p.span_len
        i32 = lambda *s: torch.zeros(s, dtype=torch.int32, device=dev)  # noqa: E731
        sc = dict(count=i32(1), pos=i32(1, 16), sel_pos=i32(1, top_c), sel_len=i32(1, top_c),
                  spans=i32(1, top_c, L), n_sel=i32(1), status=i32(1))
        tr = {} if self.trace is not None else None
        host = lambda t: t.detach().cpu().numpy().copy()  # noqa: E731
        if tr is not None:
            tr["scan_in"] = dict(tokens=host(self.buf[:self.n]), k_star=host(self.k_star), gate_ok=host(self.ok),
                                 scores=host(self.scores[:self.n]), pos_cap=16)
        if self.retrieval == "index":
            # the previous step's committed tokens join the index (Algorithm 1's update), then the query
            rs.rs_match_index_append(self.buf, tok_off, 1, self.t.V, self.idx_t, self.idx, self.idx_status)
            rs.rs_match_scan_indexed(self.buf, tok_off, 1, self.k_star, self.ok, self.scores, p, 16, sc["count"],
                                     sc["pos"], sc["sel_pos"], sc["sel_len"], sc["spans"], sc["n_sel"], sc["status"],
                                     self.t.V, self.idx_t, self.idx)
        else:
            rs.rs_match_scan(self.buf, tok_off, 1, self.k_star, self.ok, self.scores, p, 16, sc["count"], sc["pos"],
                             sc["sel_pos"], sc["sel_len"], sc["spans"], sc["n_sel"], sc["status"])
        if tr is not None:
            tr["scan_out"] = {k: host(v) for k, v in sc.items()}
        # 3. model drafts, then the chains under the root
        toks, par = self._draft_tree(root)
        source = [0] + [1] * (len(toks) - 1)
        chain = [-1] * len(toks)
        n_sel = int(sc["n_sel"][0])
        sel_len, spans = sc["sel_len"][0].cpu().numpy(), sc["spans"][0].cpu().numpy()
        for c in range(n_sel):
            prev = 0
            for j in range(int(sel_len[c])):
                toks.append(int(spans[c, j]))
                par.append(prev)
                source.append(2)
                chain.append(c)
                prev = len(toks) - 1
        N = len(toks)
        # 4. verification
        t_tok = torch.tensor(toks, dtype=torch.int32, device=dev)
        t_par = torch.tensor(par, dtype=torch.int32, device=dev)
        logits = self.t.forward_tree(self.tc, t_tok.long(), t_par, self.ws_attn).float().contiguous()
        node_off = torch.tensor([0, N], dtype=torch.int32, device=dev)
        o = dict(argmax=i32(N), topk=i32(N, p.beta), lse=torch.zeros(N, device=dev),
                 p_tok=torch.zeros(N, device=dev), entropy=torch.zeros(N, device=dev), acc_len=i32(1),
                 acc_nodes=i32(1, self.acc_cap), bonus=i32(1), winner=i32(1),
                 commit=torch.zeros(N, dtype=torch.uint8, device=dev), status=i32(1))
        ws = torch.empty(max(rs.rs_accept_workspace_size(N, self.t.V, p.beta), 256), dtype=torch.uint8, device=dev)
        if tr is not None:
            tr["accept_in"] = dict(logits=host(logits), tokens=np.array(toks, np.int32), parents=np.array(par, np.int32),
                                   source=np.array(source, np.uint8), chain=np.array(chain, np.int8),
                                   sel_pos=host(sc["sel_pos"]), scores=host(self.scores[:self.n]),
                                   acc_cap=self.acc_cap)
        rs.rs_accept(logits, N, self.t.V, node_off, 1, t_tok, t_par,
                     torch.tensor(source, dtype=torch.uint8, device=dev),
                     torch.tensor(chain, dtype=torch.int8, device=dev), sc["sel_pos"], tok_off, p, self.acc_cap,
                     o["argmax"], o["topk"], o["lse"], o["p_tok"], o["entropy"], o["acc_len"], o["acc_nodes"],
                     o["bonus"], o["winner"], o["commit"], self.scores, o["status"], ws)
        if tr is not None:
            tr["accept_out"] = dict({k: host(v) for k, v in o.items()}, scores=host(self.scores[:self.n]))
        # 5. commit: accepted tokens + bonus; K/V of the root and accepted slots into the prefix
        acc = o["acc_nodes"][0, :int(o["acc_len"][0])].cpu().numpy().tolist()
        argmax = o["argmax"].cpu().numpy()
        new = [toks[a] for a in acc] + [int(o["bonus"][0])]
        self.buf[self.n:self.n + len(new)] = torch.tensor(new, dtype=torch.int32, device=dev)
        self.t.commit(self.tc, [0] + acc)
        # the draft cache learns the committed tokens (root + accepted) as a chain
        committed = torch.tensor([root] + [toks[a] for a in acc], dtype=torch.int64, device=dev)
        self.dr.forward_tree(self.dc, committed, self._chain_parents(committed.numel()), self.ws_attn)
        self.dr.commit(self.dc, list(range(committed.numel())))
        self.n += len(new)
        # 1. (next step's) trigger from this verify's committed rows
        if tr is not None:
            tr["gate_in"] = dict(hist=host(self.hist), hist_n=host(self.hist_n))
        rs.rs_entropy_gate_rows(o["entropy"], node_off, o["commit"], 1, p, self.hist, self.hist_n,
                                self.k_star, self.h_best, self.ok)
        if tr is not None:
            tr["gate_out"] = dict(hist=host(self.hist), hist_n=host(self.hist_n), k_star=host(self.k_star),
                                  h_best=host(self.h_best), ok=host(self.ok))
            self.trace.append(tr)
        st = self.stats
        st["steps"] += 1
        st["emitted"] += len(new)
        st["triggered"] += int(n_sel > 0)
        w = int(o["winner"][0])
        st["model_wins"] += int(w == -1)
        st["retrieval_wins"] += int(w >= 0)
        st["relaxed"] += sum(1 for a in acc if toks[a] != argmax[par[a]])
        return new

    def generate(self, n_new):
        out = []
        while len(out) < n_new and self.n + 260 < self.cap:
            out += self.step()
        return np.array(out[:n_new], np.int64)


def make_prompt(V, n, seed=0, seg=32, copy_prob=0.5):
    """Synthetic prompt: segments of fresh tokens, half of them copies of earlier ones."""
    rng = np.random.default_rng(seed)
    out = []
    while len(out) < n:
        if out and rng.random() < copy_prob:
            a = int(rng.integers(0, max(1, len(out) - seg)))
            out += out[a:a + seg]
        else:
            out += rng.integers(0, V, seg).tolist()
    return np.array(out[:n], np.int32)


def model_prompt(model, n, seed=0):
    """The model's own greedy text from a random 16-token seed: like a model
    re-reading what it wrote, it repeats itself, which is what retrieval uses
    (this random model mostly follows a token with the same successor as the
    last time it saw it)."""
    start = np.random.default_rng(seed).integers(0, model.V, 16).astype(np.int32)
    return np.concatenate([start, greedy_reference(model, start, n - 16)]).astype(np.int32)


def run(tau, m, n_new=256, prompt_len=512, seed=0, noise=0.1):
    target = TinyLM(seed=seed)
    draft = TinyLM(seed=seed + 1, base=target, noise=noise)
    p = rs.params(tau=tau, m=m, span_len=8)
    loop = SpecLoop(target, draft, model_prompt(target, prompt_len, seed), p)
    loop.generate(n_new)
    s = loop.stats
    return dict(tau=tau, m=m, steps=s["steps"], mean_tokens_per_step=s["emitted"] / max(1, s["steps"]),
                trigger_rate=s["triggered"] / max(1, s["steps"]), retrieval_wins=s["retrieval_wins"],
                model_wins=s["model_wins"], non_greedy_tokens=s["relaxed"])


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--sweep", action="store_true", help="tau in {0,1,2,3} x m in {1,2,3}")
    ap.add_argument("--tokens", type=int, default=256)
    ap.add_argument("--seeds", type=int, default=1)
    args = ap.parse_args()
    taus, ms = ([0.0, 1.0, 2.0, 3.0], [1, 2, 3]) if args.sweep else ([3.0], [2])
    for tau in taus:
        for m in ms:
            runs = [run(tau, m, n_new=args.tokens, seed=s) for s in range(args.seeds)]
            steps = sum(r["steps"] for r in runs)
            row = dict(tau=tau, m=m, seeds=args.seeds, tokens=args.tokens * args.seeds, steps=steps,
                       mean_tokens_per_step=round(sum(r["mean_tokens_per_step"] * r["steps"] for r in runs) / steps, 3),
                       trigger_rate=round(sum(r["trigger_rate"] * r["steps"] for r in runs) / steps, 3),
                       retrieval_win_rate=round(sum(r["retrieval_wins"] for r in runs) / steps, 3),
                       non_greedy_per_100=round(100.0 * sum(r["non_greedy_tokens"] for r in runs)
                                                / (args.tokens * args.seeds), 2))
            print(json.dumps(row), flush=True)


if __name__ == "__main__":
    main()
