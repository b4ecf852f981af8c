"""Retrieval on long buffers: rs_match_scan (O(t) per query) against
rs_match_scan_indexed (O(occurrences of the key's last token) per query, after
an O(t) rs_match_index_build).

``python -m paper_2511_01282_gb300.retrieval_bench`` prints one JSON line per
buffer length: device time of one query call (CUDA graph of 20 calls, CUDA
events) for the scan and the index, and of one index build.  The calls run back
to back, so buffers that fit in the L2 are read from it: the times compare the
two methods rather than give the cold cost of a query.  Buffers are
synthetic (seeded): V = 32000, segments of 8-64 tokens of which 30 % copy an
earlier segment, scores uniform in [0, 1), key lengths 1-3.
"""
import argparse
import json

import numpy as np
import torch

from . import respec as rs


def make_buffers(B, t, V=32000, seed=0):
    rng = np.random.default_rng(seed)
    bufs = []
    for _ in range(B):
        out = []
        while len(out) < t:
            n = int(rng.integers(8, 65))
            if out and rng.random() < 0.3:
                a = int(rng.integers(0, max(1, len(out) - n)))
                out += out[a:a + n]
            else:
                out += rng.integers(0, V, n).tolist()
        bufs.append(np.array(out[:t], np.int32))
    return bufs


def time_graph(fn, n=20):
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        fn(s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            for _ in range(n):
                fn(s)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        g.replay()
        a.record(s)
        g.replay()
        b.record(s)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / n * 1e3


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--B", type=int, default=4)
    ap.add_argument("--lengths", default="32768,262144,1048576,4194304")
    args = ap.parse_args()
    V, B = 32000, args.B
    p = rs.params()
    for t in [int(x) for x in args.lengths.split(",")]:
        bufs = make_buffers(B, t, V)
        tok_off = torch.tensor(np.concatenate([[0], np.cumsum([len(x) for x in bufs])]), dtype=torch.int64,
                               device="cuda")
        tokens = torch.from_numpy(np.concatenate(bufs)).cuda()
        scores = torch.rand(tokens.numel(), device="cuda")
        ks = torch.tensor([1, 2, 3, 2][:B] * (B // 4 + 1), dtype=torch.int32, device="cuda")[:B].contiguous()
        t_total = tokens.numel()
        idx = torch.empty(rs.rs_match_index_bytes(B, V, t_total), dtype=torch.uint8, device="cuda")
        z = lambda *s: torch.zeros(s, dtype=torch.int32, device="cuda")  # noqa: E731
        o1 = [z(B), z(B, 1024), z(B, p.top_c), z(B, p.top_c), z(B, p.top_c, p.span_len), z(B), z(B)]
        o2 = [z(B), z(B, 1024), z(B, p.top_c), z(B, p.top_c), z(B, p.top_c, p.span_len), z(B), z(B)]
        scan_us = time_graph(lambda s: rs.rs_match_scan(tokens, tok_off, B, ks, None, scores, p, 1024, *o1,
                                                        stream=s))
        build_us = time_graph(lambda s: rs.rs_match_index_build(tokens, tok_off, B, V, t_total, idx, stream=s), n=3)
        idx_us = time_graph(lambda s: rs.rs_match_scan_indexed(tokens, tok_off, B, ks, None, scores, p, 1024,
                                                               *o2, V, t_total, idx, stream=s))
        same = all(bool((a == b).all()) for a, b in zip(o1, o2))
        print(json.dumps(dict(B=B, t=t, V=V, scan_us=round(scan_us, 2), indexed_us=round(idx_us, 2),
                              build_us=round(build_us, 1), count=o1[0].tolist(), same_outputs=same)),
              flush=True)


if __name__ == "__main__":
    main()
