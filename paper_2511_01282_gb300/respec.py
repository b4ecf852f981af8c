"""Thin ctypes binding of ``librespec.so`` (declared in ``include/respec.h``).

Argument marshalling only: every function here has the name and argument
order of its C entry point, turns torch tensors into device pointers, calls
the library and raises ``RespecError`` with the library's message when the
call returns a non-zero status.  All computation happens in the CUDA
kernels; there is no fallback of any kind -- without the compiled library
(or without a GPU) every call fails.
"""
import ctypes as C
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "librespec.so")

RS_OK, RS_ERR_INVALID_ARG, RS_ERR_UNSUPPORTED, RS_ERR_CAPACITY, RS_ERR_CUDA = range(5)
RS_ST_BAD_TREE, RS_ST_TRUNCATED, RS_ST_BAD_POS, RS_ST_TOO_LARGE, RS_ST_TIMEOUT = 1, 2, 4, 8, 16
RS_ST_BAD_OFFSET = 32
RS_MAX_L, RS_MAX_TOPC, RS_MAX_SPAN, RS_MAX_BETA, RS_MAX_NODES = 8, 8, 256, 16, 256


class RespecError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("rs_status %d: %s" % (status, msg))
        self.status = status


class rs_params(C.Structure):
    _fields_ = [("l", C.c_int), ("lambda_e", C.c_float), ("theta_entropy", C.c_float),
                ("alpha", C.c_float), ("theta_score", C.c_float), ("top_c", C.c_int),
                ("span_len", C.c_int), ("beta", C.c_int), ("tau", C.c_float), ("phi", C.c_int),
                ("m", C.c_int)]


DEFAULT_PARAMS = dict(l=3, lambda_e=0.5, theta_entropy=1.5, alpha=0.3, theta_score=0.3, top_c=3,
                      span_len=8, beta=5, tau=3.0, phi=2, m=2)


def params(**kw):
    d = dict(DEFAULT_PARAMS)
    d.update(kw)
    return rs_params(**d)


_lib = None
_P = C.c_void_p
_SIGS = {
    "rs_last_error": (C.c_char_p, []),
    "rs_version": (C.c_char_p, []),
    "rs_launch_count": (C.c_uint64, []),
    "rs_entropy_gate_workspace_size": (C.c_size_t, [C.c_int, C.c_int]),
    "rs_entropy_gate": (C.c_int, [_P, C.c_int, C.c_int, _P, _P, C.c_int, rs_params,
                                  _P, _P, _P, _P, _P, _P, _P, C.c_size_t, _P]),
    "rs_entropy_gate_noalloc": (C.c_int, [_P, C.c_int, C.c_int, _P, _P, C.c_int, rs_params,
                                          _P, _P, _P, _P, _P, _P, _P]),
    "rs_match_scan_workspace_size": (C.c_size_t, [C.c_int]),
    "rs_match_scan": (C.c_int, [_P, _P, C.c_int, _P, _P, _P, rs_params, C.c_int,
                                _P, _P, _P, _P, _P, _P, _P, _P, C.c_size_t, _P]),
    "rs_tree_verify_attn_workspace_size": (C.c_size_t, [C.c_int] * 5),
    "rs_tree_verify_attn": (C.c_int, [_P, _P, _P, C.c_int64, _P, _P, _P, _P, C.c_int, C.c_int,
                                      C.c_int, C.c_int, C.c_int, C.c_float, _P, _P, _P, _P,
                                      C.c_size_t, _P]),
    "rs_accept_workspace_size": (C.c_size_t, [C.c_int, C.c_int, C.c_int]),
    "rs_accept": (C.c_int, [_P, C.c_int, C.c_int, _P, C.c_int, _P, _P, _P, _P, _P, _P, rs_params,
                            C.c_int, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, C.c_size_t,
                            _P]),
    "rs_match_index_bytes": (C.c_size_t, [C.c_int, C.c_int, C.c_int64]),
    "rs_match_index_build": (C.c_int, [_P, _P, C.c_int, C.c_int, C.c_int64, _P, C.c_size_t, _P]),
    "rs_match_index_append": (C.c_int, [_P, _P, C.c_int, C.c_int, C.c_int64, _P, C.c_size_t, _P, _P]),
    "rs_match_scan_indexed": (C.c_int, [_P, _P, C.c_int, _P, _P, _P, rs_params, C.c_int] + [_P] * 7
                              + [C.c_int, C.c_int64, _P, C.c_size_t, _P]),
    "rs_tree_sample_workspace_size": (C.c_size_t, [C.c_int, C.c_int]),
    "rs_tree_sample": (C.c_int, [_P, C.c_int, C.c_int, _P, C.c_int, _P, _P, _P, C.c_float, _P, C.c_int,
                                 _P, _P, _P, _P, _P, _P, C.c_size_t, _P]),
    "rs_entropy_gate_rows": (C.c_int, [_P, _P, _P, C.c_int, rs_params, _P, _P, _P, _P, _P, _P]),
}


def lib():
    """Load the library (built in-tree by ``build.build()``); never falls back."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("librespec.so is not built: run paper_2511_01282_gb300.build.build() "
                               "(or __graft_entry__.build())")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def exported_symbols():
    return list(_SIGS)


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor, got one on %s" % t.device)
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status):
    if status != RS_OK:
        raise RespecError(status, lib().rs_last_error().decode())


def rs_last_error():
    return lib().rs_last_error().decode()


def rs_version():
    return lib().rs_version().decode()


def rs_launch_count():
    return int(lib().rs_launch_count())


def _ws(ws):
    if ws is None:
        return None, 0
    return _ptr(ws), ws.numel() * ws.element_size()


# ------------------------------------------------------------ entry points
def rs_entropy_gate_workspace_size(R, V):
    return int(lib().rs_entropy_gate_workspace_size(R, V))


def rs_entropy_gate(logits, R, V, row_off, row_commit, B, p, hist, hist_n, entropy, k_star,
                    h_best, entropy_ok, workspace, stream=None):
    wp, wb = _ws(workspace)
    _check(lib().rs_entropy_gate(_ptr(logits), R, V, _ptr(row_off), _ptr(row_commit), B, p,
                                 _ptr(hist), _ptr(hist_n), _ptr(entropy), _ptr(k_star),
                                 _ptr(h_best), _ptr(entropy_ok), wp, wb, _stream(stream)))


RS_GATE_NOALLOC_MAX_PARTIALS = 65536


def rs_entropy_gate_noalloc(logits, R, V, row_off, row_commit, B, p, hist, hist_n, entropy, k_star,
                            h_best, entropy_ok, stream=None):
    """rs_entropy_gate with the library's fixed scratch array instead of a
    caller workspace (for callers that cannot allocate device memory)."""
    _check(lib().rs_entropy_gate_noalloc(_ptr(logits), R, V, _ptr(row_off), _ptr(row_commit), B, p,
                                         _ptr(hist), _ptr(hist_n), _ptr(entropy), _ptr(k_star),
                                         _ptr(h_best), _ptr(entropy_ok), _stream(stream)))


def rs_match_scan_workspace_size(B):
    return int(lib().rs_match_scan_workspace_size(B))


def rs_match_scan(tokens, tok_off, B, k_star, gate_ok, scores, p, pos_cap, count, pos, sel_pos,
                  sel_len, spans, n_sel, status, workspace=None, stream=None):
    wp, wb = _ws(workspace)
    _check(lib().rs_match_scan(_ptr(tokens), _ptr(tok_off), B, _ptr(k_star), _ptr(gate_ok),
                               _ptr(scores), p, pos_cap, _ptr(count), _ptr(pos), _ptr(sel_pos),
                               _ptr(sel_len), _ptr(spans), _ptr(n_sel), _ptr(status), wp, wb,
                               _stream(stream)))


def rs_tree_verify_attn_workspace_size(B, R, Hq, Hkv, D):
    return int(lib().rs_tree_verify_attn_workspace_size(B, R, Hq, Hkv, D))


def rs_tree_verify_attn(q, k, v, kv_rows, kv_off, ctx_len, node_off, parents, B, R, Hq, Hkv, D,
                        scale, out, lse, status, workspace, stream=None):
    wp, wb = _ws(workspace)
    _check(lib().rs_tree_verify_attn(_ptr(q), _ptr(k), _ptr(v), kv_rows, _ptr(kv_off),
                                     _ptr(ctx_len), _ptr(node_off), _ptr(parents), B, R, Hq, Hkv,
                                     D, scale, _ptr(out), _ptr(lse), _ptr(status), wp, wb,
                                     _stream(stream)))


def rs_accept_workspace_size(R, V, beta):
    return int(lib().rs_accept_workspace_size(R, V, beta))


def rs_match_index_bytes(B, V, t_total):
    return int(lib().rs_match_index_bytes(B, V, t_total))


def rs_match_index_build(tokens, tok_off, B, V, t_total, index, stream=None):
    _check(lib().rs_match_index_build(_ptr(tokens), _ptr(tok_off), B, V, t_total, _ptr(index),
                                      index.numel() * index.element_size(), _stream(stream)))


def rs_match_index_append(tokens, tok_off, B, V, t_total, index, status=None, stream=None):
    _check(lib().rs_match_index_append(_ptr(tokens), _ptr(tok_off), B, V, t_total, _ptr(index),
                                       index.numel() * index.element_size(), _ptr(status), _stream(stream)))


def rs_match_scan_indexed(tokens, tok_off, B, k_star, gate_ok, scores, p, pos_cap, count, pos, sel_pos,
                          sel_len, spans, n_sel, status, V, t_total, index, stream=None):
    _check(lib().rs_match_scan_indexed(_ptr(tokens), _ptr(tok_off), B, _ptr(k_star), _ptr(gate_ok),
                                       _ptr(scores), p, pos_cap, _ptr(count), _ptr(pos), _ptr(sel_pos),
                                       _ptr(sel_len), _ptr(spans), _ptr(n_sel), _ptr(status), V, t_total,
                                       _ptr(index), index.numel() * index.element_size(),
                                       _stream(stream)))


def rs_tree_sample_workspace_size(R, V):
    return int(lib().rs_tree_sample_workspace_size(R, V))


def rs_tree_sample(logits, R, V, node_off, B, tokens, parents, source, temperature, uniforms,
                   acc_cap, draw, acc_len, acc_nodes, bonus, status, workspace, stream=None):
    wp, wb = _ws(workspace)
    _check(lib().rs_tree_sample(_ptr(logits), R, V, _ptr(node_off), B, _ptr(tokens),
                                _ptr(parents), _ptr(source), float(temperature), _ptr(uniforms),
                                acc_cap, _ptr(draw), _ptr(acc_len), _ptr(acc_nodes), _ptr(bonus),
                                _ptr(status), wp, wb, _stream(stream)))


def rs_accept(logits, R, V, node_off, B, tokens, parents, source, chain, sel_pos, tok_off, p,
              acc_cap, argmax, topk, lse, p_tok, entropy, acc_len, acc_nodes, bonus, winner, commit,
              scores, status, workspace, stream=None):
    wp, wb = _ws(workspace)
    _check(lib().rs_accept(_ptr(logits), R, V, _ptr(node_off), B, _ptr(tokens), _ptr(parents),
                           _ptr(source), _ptr(chain), _ptr(sel_pos), _ptr(tok_off), p, acc_cap,
                           _ptr(argmax), _ptr(topk), _ptr(lse), _ptr(p_tok), _ptr(entropy),
                           _ptr(acc_len), _ptr(acc_nodes), _ptr(bonus), _ptr(winner),
                           _ptr(commit), _ptr(scores), _ptr(status), wp, wb, _stream(stream)))


def rs_entropy_gate_rows(entropy, row_off, row_commit, B, p, hist, hist_n, k_star, h_best,
                         entropy_ok, stream=None):
    _check(lib().rs_entropy_gate_rows(_ptr(entropy), _ptr(row_off), _ptr(row_commit), B, p,
                                      _ptr(hist), _ptr(hist_n), _ptr(k_star), _ptr(h_best),
                                      _ptr(entropy_ok), _stream(stream)))
