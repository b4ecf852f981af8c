"""Plain fp64 CPU oracle of the ReSpec verify-and-draft step (ctypes wrapper).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library: the C sources here restate the paper's definitions
(Section 3.2.1 Eq. 1-3, Section 3.3, Section 3.4 Eq. 6-7, Eq. 4-5, Algorithm 1)
and this module only marshals numpy arrays into them.

Every function takes host numpy arrays and returns a dict of numpy arrays.
Floating-point parameters that the product receives as fp32 should be passed
here already rounded to fp32 (e.g. ``float(np.float32(x))``) so both sides see
the same value.
"""
import ctypes as C
import os

import numpy as np

from . import build as _build

_lib = None


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = C.CDLL(path)
        P = C.c_void_p
        L.rsref_row_entropy.restype = C.c_double
        L.rsref_row_entropy.argtypes = [P, C.c_long]
        L.rsref_entropy_rows.restype = None
        L.rsref_entropy_rows.argtypes = [P, C.c_long, C.c_long, P]
        L.rsref_gate.restype = None
        L.rsref_gate.argtypes = [P, P, P, C.c_int, C.c_int, C.c_double, C.c_double,
                                 P, P, P, P, P]
        L.rsref_match_scan.restype = C.c_int
        L.rsref_match_scan.argtypes = [P, P, C.c_int, P, P, P, C.c_double,
                                       C.c_int, C.c_int, C.c_int] + [P] * 7
        L.rsref_tree_attn.restype = C.c_int
        L.rsref_tree_attn.argtypes = [P, P, P, P, P, P, P, C.c_int, C.c_int, C.c_int,
                                      C.c_int, C.c_double, C.c_long, P, P, P, P]
        L.rsref_accept.restype = None
        L.rsref_accept.argtypes = ([P, C.c_long, P, C.c_int, P, P, P, P, P, C.c_int, P,
                                    C.c_int, C.c_double, C.c_int, C.c_int, C.c_double,
                                    C.c_int] + [P] * 11)
        L.rsref_sample_row.restype = C.c_int
        L.rsref_sample_row.argtypes = [P, C.c_long, C.c_double, C.c_double]
        L.rsref_tree_sample.restype = None
        L.rsref_tree_sample.argtypes = ([P, C.c_long, P, C.c_int, P, P, P, C.c_double, P, C.c_int]
                                        + [P] * 5)
        _lib = L
    return _lib


def _c(a, dtype):
    """Contiguous array of the given dtype (a copy only when needed)."""
    return np.ascontiguousarray(a, dtype=dtype)


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


# ---------------------------------------------------------------- entropy
def row_entropy(z):
    """Eq. 1 inner term for one row of logits (nats)."""
    z = _c(z, np.float32)
    return lib().rsref_row_entropy(_p(z), z.size)


def entropy_rows(logits):
    """Per-row entropy (nats) of an [R, V] fp32 logits matrix."""
    logits = _c(logits, np.float32)
    R, V = logits.shape
    H = np.empty(R, np.float64)
    lib().rsref_entropy_rows(_p(logits), R, V, _p(H))
    return H


def gate(H, row_off, row_commit, hist, hist_n, l, lambda_e, theta):
    """Section 3.2.1 (entropy, confidence score, key selection, trigger decision; Algorithm 1's triggering) on given row entropies.

    ``hist`` [B, l] (oldest first) and ``hist_n`` [B] are copied, updated and
    returned; the inputs are left untouched.
    """
    H = _c(H, np.float64)
    row_off = _c(row_off, np.int64)
    row_commit = _c(row_commit, np.uint8)
    B = row_off.size - 1
    hist = np.array(hist, dtype=np.float64).reshape(B, l).copy()
    hist_n = np.array(hist_n, dtype=np.int32).copy()
    k_star = np.empty(B, np.int32)
    h_best = np.empty(B, np.float64)
    ok = np.empty(B, np.uint8)
    lib().rsref_gate(_p(H), _p(row_off), _p(row_commit), B, l, lambda_e, theta,
                     _p(hist), _p(hist_n), _p(k_star), _p(h_best), _p(ok))
    return dict(hist=hist, hist_n=hist_n, k_star=k_star, h_best=h_best, ok=ok)


# ---------------------------------------------------------------- match scan
def match_scan(tokens, tok_off, k_star, scores, theta_score, top_c, span_len, pos_cap,
               gate_ok=None):
    """Section 3.3 retrieval + selection (Algorithm 1's retrieval)."""
    tokens = _c(tokens, np.int32)
    tok_off = _c(tok_off, np.int64)
    k_star = _c(k_star, np.int32)
    scores = _c(scores, np.float32)
    B = tok_off.size - 1
    go = None if gate_ok is None else _c(gate_ok, np.uint8)
    out = dict(count=np.empty(B, np.int32),
               pos=np.empty((B, pos_cap), np.int32),
               sel_pos=np.empty((B, top_c), np.int32),
               sel_len=np.empty((B, top_c), np.int32),
               spans=np.empty((B, top_c, span_len), np.int32),
               n_sel=np.empty(B, np.int32),
               status=np.empty(B, np.int32))
    lib().rsref_match_scan(_p(tokens), _p(tok_off), B, _p(k_star), _p(go), _p(scores),
                           theta_score, top_c, span_len, pos_cap,
                           _p(out["count"]), _p(out["pos"]), _p(out["sel_pos"]),
                           _p(out["sel_len"]), _p(out["spans"]), _p(out["n_sel"]),
                           _p(out["status"]))
    return out


# ---------------------------------------------------------------- attention
def tree_attn(q, k, v, kv_off, ctx_len, node_off, parents, Hq, Hkv, D, scale,
              rows=None):
    """Tree-verification attention for (node, head) pairs.

    q: [R, Hq, D] bf16 bits (uint16); k, v: [T, Hkv, D] bf16 bits.
    ``rows``: None for every (node, head), else an iterable of (node, head).
    Returns dict(out [n, D] f64, lse [n] f64, rows [n, 2], rc).
    """
    q = _c(q, np.uint16)
    k = _c(k, np.uint16)
    v = _c(v, np.uint16)
    kv_off = _c(kv_off, np.int64)
    ctx_len = _c(ctx_len, np.int32)
    node_off = _c(node_off, np.int32)
    parents = _c(parents, np.int32)
    B = node_off.size - 1
    R = int(node_off[-1])
    if rows is None:
        rr = np.stack(np.meshgrid(np.arange(R), np.arange(Hq), indexing="ij"), -1).reshape(-1, 2)
    else:
        rr = np.asarray(list(rows), dtype=np.int64).reshape(-1, 2)
    row_node = _c(rr[:, 0], np.int64)
    row_head = _c(rr[:, 1], np.int32)
    n = rr.shape[0]
    out = np.zeros((n, D), np.float64)
    lse = np.zeros(n, np.float64)
    rc = lib().rsref_tree_attn(_p(q), _p(k), _p(v), _p(kv_off), _p(ctx_len), _p(node_off),
                               _p(parents), B, Hq, Hkv, D, scale, n, _p(row_node),
                               _p(row_head), _p(out), _p(lse))
    return dict(out=out, lse=lse, rows=rr, rc=rc)


# ---------------------------------------------------------------- accept
def accept(logits, node_off, tokens, parents, source, chain, sel_pos, tok_off, scores,
           beta, tau, phi, m, alpha, acc_cap):
    """Section 3.4 verification + longest path + Eq. 4-5 EMA update.

    ``scores`` is copied, updated and returned (fp32 storage).
    """
    logits = _c(logits, np.float32)
    R, V = logits.shape
    node_off = _c(node_off, np.int32)
    B = node_off.size - 1
    tokens = _c(tokens, np.int32)
    parents = _c(parents, np.int32)
    source = _c(source, np.uint8)
    chain = _c(chain, np.int8)
    sel_pos = _c(sel_pos, np.int32).reshape(B, -1)
    top_c = sel_pos.shape[1]
    tok_off = _c(tok_off, np.int64)
    scores = np.array(scores, dtype=np.float32).copy()
    out = dict(argmax=np.empty(R, np.int32),
               topk=np.empty((R, beta), np.int32),
               lse=np.empty(R, np.float64),
               p_tok=np.empty(R, np.float64),
               acc_len=np.empty(B, np.int32),
               acc_nodes=np.empty((B, acc_cap), np.int32),
               bonus=np.empty(B, np.int32),
               winner=np.empty(B, np.int32),
               commit=np.empty(R, np.uint8),
               status=np.empty(B, np.int32))
    sel_pos = np.ascontiguousarray(sel_pos)
    lib().rsref_accept(_p(logits), V, _p(node_off), B, _p(tokens), _p(parents), _p(source),
                       _p(chain), _p(sel_pos), top_c, _p(tok_off), beta, tau, phi, m, alpha,
                       acc_cap, _p(out["argmax"]), _p(out["topk"]), _p(out["lse"]),
                       _p(out["p_tok"]), _p(out["acc_len"]), _p(out["acc_nodes"]),
                       _p(out["bonus"]), _p(out["winner"]), _p(out["commit"]), _p(scores),
                       _p(out["status"]))
    out["scores"] = scores
    return out


# ---------------------------------------------------------------- sampling
def sample_row(z, T, u):
    """Section 3.4 drafter outputs: the inverse-CDF draw (token-id order) from softmax(z/T)."""
    z = _c(z, np.float32)
    return int(lib().rsref_sample_row(_p(z), z.size, float(T), float(u)))


def tree_sample(logits, node_off, tokens, parents, source, T, u, acc_cap):
    """Per-row draws and the lossless walk over the model-drafted nodes."""
    logits = _c(logits, np.float32)
    R, V = logits.shape
    node_off = _c(node_off, np.int32)
    B = node_off.size - 1
    u = _c(u, np.float64)
    out = dict(draw=np.empty(R, np.int32), acc_len=np.empty(B, np.int32),
               acc_nodes=np.empty((B, acc_cap), np.int32), bonus=np.empty(B, np.int32),
               status=np.empty(B, np.int32))
    lib().rsref_tree_sample(_p(logits), V, _p(node_off), B, _p(_c(tokens, np.int32)),
                            _p(_c(parents, np.int32)), _p(_c(source, np.uint8)), float(T), _p(u),
                            acc_cap, _p(out["draw"]), _p(out["acc_len"]), _p(out["acc_nodes"]),
                            _p(out["bonus"]), _p(out["status"]))
    return out


ST_BAD_TREE = 1
ST_TRUNCATED = 2
ST_BAD_POS = 4
