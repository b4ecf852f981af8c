"""C-ABI library checks that need no GPU: it builds, loads, exports every
symbol ``include/respec.h`` declares, and rejects bad host arguments before
launching anything.  Also checks that the oracle and the CUDA library share
no source."""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "respec.h")


@pytest.fixture(scope="module")
def rs():
    from paper_2511_01282_gb300 import build
    build.build()
    from paper_2511_01282_gb300 import respec
    respec.lib()
    return respec


def _declared():
    txt = open(HEADER).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(rs_[a-z_]+)\s*\(", txt)))


def test_header_declares_the_four_calls():
    names = _declared()
    for n in ("rs_entropy_gate", "rs_match_scan", "rs_tree_verify_attn", "rs_accept"):
        assert n in names and n + "_workspace_size" in names


def test_every_declared_symbol_is_exported(rs):
    out = subprocess.run(["nm", "-D", "--defined-only", rs.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (rs_\w+)", out))
    missing = [n for n in _declared() if n not in exported]
    assert not missing, missing
    # and the binding knows each of them
    assert sorted(rs.exported_symbols()) == sorted(_declared())


def test_library_identifies_itself(rs):
    assert "sm_103a" in rs.rs_version()
    assert rs.rs_launch_count() >= 0


def test_params_struct_layout_matches_header(rs):
    # 11 four-byte fields, no padding
    assert C.sizeof(rs.rs_params) == 44
    txt = open(HEADER).read()
    body = re.search(r"typedef struct \{(.*?)\} rs_params;", txt, re.S).group(1)
    fields = re.findall(r"\b(int|float)\s+([a-z_]+)\s*;", re.sub(r"/\*.*?\*/", "", body, flags=re.S))
    assert [f for _, f in fields] == [f for f, _ in rs.rs_params._fields_]


def test_workspace_sizes_are_host_computable(rs):
    assert rs.rs_entropy_gate_workspace_size(145, 128256) >= 145 * 16 * 12
    assert rs.rs_accept_workspace_size(145, 128256, 5) >= 145 * 16 * 5 * 8
    assert rs.rs_match_scan_workspace_size(4) >= 0
    assert rs.rs_entropy_gate_workspace_size(-1, 10) == 0
    assert rs.rs_tree_sample_workspace_size(145, 128256) >= 145 * 16 * 8
    assert rs.rs_tree_sample_workspace_size(3, 0) == 0
    assert rs.rs_match_index_bytes(4, 32000, 131072) >= 131072 * 4 + 4 * 32002 * 4
    assert rs.rs_match_index_bytes(4, 0, 10) == 0


def _fake(n=1):
    return C.c_void_p(0x10000)  # never dereferenced: every call below fails its host checks


def test_bad_arguments_fail_before_launch(rs):
    L = rs.lib()
    p = rs.params()
    f = _fake()
    n_launch = rs.rs_launch_count()
    # rs_entropy_gate: l out of range
    bad = rs.params(l=0)
    st = L.rs_entropy_gate(f, 1, 10, f, f, 1, bad, f, f, f, f, f, f, f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG and "l=0" in rs.rs_last_error()
    # V = 0
    st = L.rs_entropy_gate(f, 1, 0, f, f, 1, p, f, f, f, f, f, f, f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG
    # workspace too small
    st = L.rs_entropy_gate(f, 4, 100000, f, f, 1, p, f, f, f, f, f, f, f, 8, None)
    assert st == rs.RS_ERR_CAPACITY and "workspace" in rs.rs_last_error()
    # rs_accept: beta above V, negative tau, null pointers
    st = L.rs_accept(f, 1, 3, f, 1, f, f, f, f, f, f, rs.params(beta=5), 4, *([f] * 12), f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG
    st = L.rs_accept(f, 1, 30, f, 1, f, f, f, f, f, f, rs.params(tau=-1.0), 4, *([f] * 12), f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG
    st = L.rs_accept(None, 1, 30, f, 1, f, f, f, f, f, f, p, 4, *([f] * 12), f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG and "null" in rs.rs_last_error()
    # rs_match_scan: top_c above the limit, span_len 0
    st = L.rs_match_scan(f, f, 1, f, None, f, rs.params(top_c=9), 4, *([f] * 7), None, 0, None)
    assert st == rs.RS_ERR_INVALID_ARG
    st = L.rs_match_scan(f, f, 1, f, None, f, rs.params(span_len=0), 4, *([f] * 7), None, 0, None)
    assert st == rs.RS_ERR_INVALID_ARG
    # rs_tree_verify_attn: unsupported head dim, GQA mismatch, misaligned K
    st = L.rs_tree_verify_attn(f, f, f, 10, f, f, f, f, 1, 1, 4, 4, 96, 0.1, f, f, f, f, 1 << 30, None)
    assert st == rs.RS_ERR_UNSUPPORTED and "96" in rs.rs_last_error()
    st = L.rs_tree_verify_attn(f, f, f, 10, f, f, f, f, 1, 1, 6, 4, 128, 0.1, f, f, f, f, 1 << 30, None)
    assert st == rs.RS_ERR_UNSUPPORTED
    st = L.rs_tree_verify_attn(f, C.c_void_p(0x10002), f, 10, f, f, f, f, 1, 1, 4, 4, 128, 0.1, f, f, f, f,
                               1 << 30, None)
    assert st == rs.RS_ERR_INVALID_ARG and "aligned" in rs.rs_last_error()
    # more requests than a call takes
    st = L.rs_tree_verify_attn(f, f, f, 10, f, f, f, f, 3841, 1, 4, 4, 128, 0.1, f, f, f, f, 1 << 30, None)
    assert st == rs.RS_ERR_INVALID_ARG and "3840" in rs.rs_last_error()
    # a KV cache whose tile count could overflow the 32-bit work split is refused
    st = L.rs_tree_verify_attn(f, f, f, (1 << 31) - 256, f, f, f, f, 1, 1, 64, 64, 128, 0.1, f, f, f, f, 1 << 30,
                               None)
    assert st == rs.RS_ERR_UNSUPPORTED and "32-bit work split" in rs.rs_last_error()
    # misaligned output rows or workspace
    st = L.rs_tree_verify_attn(f, f, f, 10, f, f, f, f, 1, 1, 4, 4, 128, 0.1, C.c_void_p(0x10004), f, f, f,
                               1 << 30, None)
    assert st == rs.RS_ERR_INVALID_ARG and "aligned" in rs.rs_last_error()
    st = L.rs_tree_verify_attn(f, f, f, 10, f, f, f, f, 1, 1, 4, 4, 128, 0.1, f, f, f, C.c_void_p(0x10008),
                               1 << 30, None)
    assert st == rs.RS_ERR_INVALID_ARG and "aligned" in rs.rs_last_error()
    # rs_tree_sample: temperature must be finite and positive; acc_cap >= 1
    for T in (0.0, -1.0, float("inf"), float("nan")):
        st = L.rs_tree_sample(f, 1, 10, f, 1, f, f, f, T, f, 4, f, f, f, f, f, f, 1 << 20, None)
        assert st == rs.RS_ERR_INVALID_ARG and "temperature" in rs.rs_last_error()
    st = L.rs_tree_sample(f, 1, 10, f, 1, f, f, f, 1.0, f, 0, f, f, f, f, f, f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG
    st = L.rs_tree_sample(f, 4, 100000, f, 1, f, f, f, 1.0, f, 4, f, f, f, f, f, f, 8, None)
    assert st == rs.RS_ERR_CAPACITY
    # index: too small a buffer for the index, bad V
    st = L.rs_match_index_build(f, f, 2, 1000, 100, f, 64, None)
    assert st == rs.RS_ERR_CAPACITY and "index" in rs.rs_last_error()
    st = L.rs_match_index_build(f, f, 2, 0, 100, f, 1 << 30, None)
    assert st == rs.RS_ERR_INVALID_ARG
    st = L.rs_match_scan_indexed(f, f, 1, f, None, f, rs.params(top_c=9), 4, *([f] * 7), 100, 10, f, 1 << 20, None)
    assert st == rs.RS_ERR_INVALID_ARG
    # nothing was launched by any of these
    assert rs.rs_launch_count() == n_launch


def test_oracle_and_library_share_no_source():
    pkg = os.path.join(ROOT, "paper_2511_01282_gb300")
    ora = os.path.join(ROOT, "oracle")
    for d, other in ((pkg, "oracle"), (ora, "paper_2511_01282_gb300")):
        for dirpath, _, files in os.walk(d):
            for fn in files:
                if fn.endswith((".c", ".h", ".cu", ".cuh", ".py")):
                    txt = open(os.path.join(dirpath, fn)).read()
                    assert not re.search(r"(import|include)[^\n]*\b%s\b" % other, txt), (fn, other)
    # the oracle restates its own constants instead of including the ABI header
    for fn in os.listdir(ora):
        if fn.endswith((".c", ".h")):
            assert "respec.h" not in open(os.path.join(ora, fn)).read()


def test_attention_form_choice_sizes_the_workspace(rs, monkeypatch):
    # the host picks the two-row-tile form (256-row partial slots) when the
    # requests average more than one 128-row tile of (node, head-in-group)
    # rows per KV head, and the workspace follows the choice: GQA 4 over 145
    # nodes (580 rows per KV head) takes it, 40 KV heads over 65 nodes per
    # request (65 rows) do not; RS_DEBUG_ATTN_FORM forces either
    ws = rs.rs_tree_verify_attn_workspace_size
    monkeypatch.delenv("RS_DEBUG_ATTN_FORM", raising=False)
    g_def, o_def = ws(1, 145, 32, 8, 128), ws(4, 260, 40, 40, 128)
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "one")
    g_one, o_one = ws(1, 145, 32, 8, 128), ws(4, 260, 40, 40, 128)
    monkeypatch.setenv("RS_DEBUG_ATTN_FORM", "pair")
    g_pair, o_pair = ws(1, 145, 32, 8, 128), ws(4, 260, 40, 40, 128)
    assert g_def == g_pair > g_one
    assert o_def == o_one < o_pair
