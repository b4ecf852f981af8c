"""One verify-and-draft step on the GPU, as the four C-ABI calls.

``VerifyStep`` owns the device buffers of one batch (inputs, outputs and the
per-call workspaces, all plain torch allocations) and enqueues, on one
stream, the calls of one step of Algorithm 1 in their data-flow order:

    trigger (rs_entropy_gate_rows on the row entropies of the last verify,
             or rs_entropy_gate on the logits)
      -> rs_match_scan (keyed by k*, gated by the trigger)
      -> rs_tree_verify_attn -> rs_accept (also emits the row entropies)

``tree_sample`` runs rs_tree_sample, the non-greedy (lossless sampling)
verification of the model drafts, and ``scan(indexed=True)`` the retrieval
from the inverted index (``build_index``), on the same buffers.  It computes
nothing itself.  Inputs come as host numpy arrays (bf16 as
uint16 bit patterns) with the layouts ``include/respec.h`` documents.
"""
import numpy as np
import torch

from . import respec as rs


def _dev(a, device):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


class VerifyStep:
    INPUTS = ("logits", "row_off", "row_commit", "hist", "hist_n", "tokens", "tok_off", "scores",
              "q", "k", "v", "kv_off", "ctx_len", "node_off", "parents", "tree_tokens", "source",
              "chain", "sel_pos")

    def __init__(self, arrays, p, Hq, Hkv, D, pos_cap=1024, acc_cap=64, device="cuda",
                 scale=None, pinned_host=False, sample_seed=0, host_blob=None):
        self.p = p
        self.Hq, self.Hkv, self.D = Hq, Hkv, D
        self.scale = float(D ** -0.5 if scale is None else scale)
        self.pos_cap, self.acc_cap = pos_cap, acc_cap
        self.device = torch.device(device)
        host = dict(arrays)
        host["row_off"] = np.asarray(host["node_off"], np.int32)
        self.host = {k: np.ascontiguousarray(host[k]) for k in self.INPUTS}
        self.B = int(self.host["node_off"].size - 1)
        self.R = int(self.host["node_off"][-1])
        self.V = int(self.host["logits"].shape[1])
        self.kv_rows = int(self.host["k"].shape[0])
        # device inputs.  With pinned_host the inputs live in one device
        # allocation (256-byte aligned views) mirrored by one pinned host
        # buffer, so that a step's upload is a single copy; host_blob shares
        # another VerifyStep's pinned buffer (same arrays).
        self.pinned_blob = None
        if pinned_host or host_blob is not None:
            layout, off = {}, 0
            for k, v in self.host.items():
                layout[k] = (off, v.nbytes, v.dtype, v.shape)
                off += -(-max(v.nbytes, 1) // 256) * 256
            if host_blob is None:
                host_blob = torch.empty(off, dtype=torch.uint8).pin_memory()
                hb = host_blob.numpy()
                for k, v in self.host.items():
                    o, n = layout[k][:2]
                    hb[o:o + n] = v.reshape(-1).view(np.uint8)
            assert host_blob.numel() == off and host_blob.is_pinned()
            self.pinned_blob = host_blob
            self.dev_blob = torch.empty(off, dtype=torch.uint8, device=self.device)
            self.dev_blob.copy_(host_blob)
            tdt = lambda dt: torch.from_numpy(np.empty(0, dt)).dtype  # noqa: E731  (as torch.from_numpy maps it)
            self.d = {k: self.dev_blob[o:o + n].view(tdt(dt)).reshape(shape)
                      for k, (o, n, dt, shape) in layout.items()}
        else:
            self.d = {k: _dev(v, self.device) for k, v in self.host.items()}
        B, R, V = self.B, self.R, self.V
        dev = self.device
        z = lambda n, dt: torch.zeros(n, dtype=dt, device=dev)  # noqa: E731
        tc, L = p.top_c, p.span_len
        self.out = dict(
            entropy=z(R, torch.float32), k_star=z(B, torch.int32), h_best=z(B, torch.float32),
            entropy_ok=z(B, torch.uint8),
            count=z(B, torch.int32), pos=z((B, pos_cap), torch.int32), sel_pos=z((B, tc), torch.int32),
            sel_len=z((B, tc), torch.int32), spans=z((B, tc, L), torch.int32), n_sel=z(B, torch.int32),
            scan_status=z(B, torch.int32),
            attn_out=z((R, Hq, D), torch.float32), attn_lse=z((R, Hq), torch.float32),
            attn_status=z(B, torch.int32),
            argmax=z(R, torch.int32), topk=z((R, p.beta), torch.int32), lse=z(R, torch.float32),
            p_tok=z(R, torch.float32), acc_entropy=z(R, torch.float32),
            acc_len=z(B, torch.int32), acc_nodes=z((B, acc_cap), torch.int32),
            bonus=z(B, torch.int32), winner=z(B, torch.int32), commit=z(R, torch.uint8),
            acc_status=z(B, torch.int32))
        self.ws = dict(
            gate=z(max(rs.rs_entropy_gate_workspace_size(R, V), 256), torch.uint8),
            scan=z(max(rs.rs_match_scan_workspace_size(B), 256), torch.uint8),
            attn=z(max(rs.rs_tree_verify_attn_workspace_size(B, R, Hq, Hkv, D), 256), torch.uint8),
            accept=z(max(rs.rs_accept_workspace_size(R, V, p.beta), 256), torch.uint8),
            sample=z(max(rs.rs_tree_sample_workspace_size(R, V), 256), torch.uint8))
        # lossless sampling of the model drafts (rs_tree_sample): one uniform per row
        gen = torch.Generator(device=dev).manual_seed(sample_seed)
        self.uniforms = torch.rand(max(R, 1), device=dev, generator=gen)
        self.sample_out = dict(draw=z(max(R, 1), torch.int32), acc_len=z(B, torch.int32),
                               acc_nodes=z((B, acc_cap), torch.int32), bonus=z(B, torch.int32),
                               status=z(B, torch.int32))

    # ------------------------------------------------------------ the calls
    def gate(self, stream=None):
        d, o = self.d, self.out
        rs.rs_entropy_gate(d["logits"], self.R, self.V, d["row_off"], d["row_commit"], self.B, self.p,
                           d["hist"], d["hist_n"], o["entropy"], o["k_star"], o["h_best"],
                           o["entropy_ok"], self.ws["gate"], stream)

    def gate_rows(self, stream=None):
        """The trigger from the row entropies the last accept produced."""
        d, o = self.d, self.out
        rs.rs_entropy_gate_rows(o["acc_entropy"], d["row_off"], d["row_commit"], self.B, self.p,
                                d["hist"], d["hist_n"], o["k_star"], o["h_best"], o["entropy_ok"],
                                stream)

    def scan(self, k_star=None, gate_ok="gate", stream=None, indexed=False):
        d, o = self.d, self.out
        ks = o["k_star"] if k_star is None else k_star
        ok = o["entropy_ok"] if gate_ok == "gate" else gate_ok
        if indexed:  # from the inverted index (build_index first)
            rs.rs_match_scan_indexed(d["tokens"], d["tok_off"], self.B, ks, ok, d["scores"], self.p, self.pos_cap,
                                     o["count"], o["pos"], o["sel_pos"], o["sel_len"], o["spans"], o["n_sel"],
                                     o["scan_status"], self.V, self.t_total, self.index, stream)
            return
        rs.rs_match_scan(d["tokens"], d["tok_off"], self.B, ks, ok, d["scores"], self.p, self.pos_cap,
                         o["count"], o["pos"], o["sel_pos"], o["sel_len"], o["spans"], o["n_sel"],
                         o["scan_status"], self.ws["scan"], stream)

    def build_index(self, stream=None):
        """Inverted index over the token buffers, for scan(indexed=True)."""
        self.t_total = int(self.host["tok_off"][-1])
        if getattr(self, "index", None) is None:
            self.index = torch.empty(rs.rs_match_index_bytes(self.B, self.V, self.t_total), dtype=torch.uint8,
                                     device=self.device)
        rs.rs_match_index_build(self.d["tokens"], self.d["tok_off"], self.B, self.V, self.t_total, self.index,
                                stream)

    def attn(self, stream=None):
        d, o = self.d, self.out
        rs.rs_tree_verify_attn(d["q"], d["k"], d["v"], self.kv_rows, d["kv_off"], d["ctx_len"],
                               d["node_off"], d["parents"], self.B, self.R, self.Hq, self.Hkv, self.D,
                               self.scale, o["attn_out"], o["attn_lse"], o["attn_status"],
                               self.ws["attn"], stream)

    def accept(self, sel_pos=None, entropy=True, stream=None):
        d, o = self.d, self.out
        sp = d["sel_pos"] if sel_pos is None else sel_pos
        rs.rs_accept(d["logits"], self.R, self.V, d["node_off"], self.B, d["tree_tokens"], d["parents"],
                     d["source"], d["chain"], sp, d["tok_off"], self.p, self.acc_cap, o["argmax"],
                     o["topk"], o["lse"], o["p_tok"], o["acc_entropy"] if entropy else None,
                     o["acc_len"], o["acc_nodes"], o["bonus"], o["winner"], o["commit"], d["scores"],
                     o["acc_status"], self.ws["accept"], stream)

    def tree_sample(self, temperature=1.0, stream=None):
        """Lossless sampling verification of the model drafts (non-greedy)."""
        d, o = self.d, self.sample_out
        rs.rs_tree_sample(d["logits"], self.R, self.V, d["node_off"], self.B, d["tree_tokens"],
                          d["parents"], d["source"], temperature, self.uniforms, self.acc_cap,
                          o["draw"], o["acc_len"], o["acc_nodes"], o["bonus"], o["status"],
                          self.ws["sample"], stream)

    def step(self, stream=None, fused=True):
        """One pass of the whole hot path.

        fused=True (steady state): the trigger uses the row entropies that the
        previous step's rs_accept computed over the verify logits, so the
        logits are read once per step; call prime() once first.
        fused=False: rs_entropy_gate reads the logits itself.
        """
        if fused:
            self.gate_rows(stream)
        else:
            self.gate(stream)
        self.scan(stream=stream)
        self.attn(stream)
        self.accept(stream=stream)

    def prime(self, stream=None):
        """Row entropies for the first fused step (one rs_accept pass)."""
        scores = self.d["scores"].clone()
        self.accept(stream=stream)
        self.d["scores"].copy_(scores)

    # ------------------------------------------------------ host round trip
    def upload(self, stream=None):
        """Copy every input from pinned host memory: one async copy on `stream`
        (needs VerifyStep(..., pinned_host=True) or a shared host_blob)."""
        if self.pinned_blob is None:
            raise RuntimeError("VerifyStep.upload: built without pinned_host=True")
        s = torch.cuda.current_stream() if stream is None else stream
        with torch.cuda.stream(s):
            self.dev_blob.copy_(self.pinned_blob, non_blocking=True)
        return self.pinned_blob.numel()

    RESULT_KEYS = ("acc_len", "acc_nodes", "bonus", "winner", "commit", "k_star", "entropy_ok",
                   "sel_pos", "n_sel")

    def download_into(self, host_bufs, stream=None):
        """Copy the step's decisions to pinned host buffers (async)."""
        s = torch.cuda.current_stream() if stream is None else stream
        n = 0
        with torch.cuda.stream(s):
            for k in self.RESULT_KEYS:
                host_bufs[k].copy_(self.out[k], non_blocking=True)
                n += self.out[k].numel() * self.out[k].element_size()
        return n

    def result_buffers(self):
        return {k: torch.empty(self.out[k].shape, dtype=self.out[k].dtype).pin_memory()
                for k in self.RESULT_KEYS}

    # ------------------------------------------- state carried across steps
    STATE_KEYS = ("hist", "hist_n", "scores")

    def reset_state(self):
        """Restore the in/out state (history, scores) to the host inputs."""
        for k in self.STATE_KEYS:
            self.d[k].copy_(torch.from_numpy(self.host[k]))

    def state(self, stream=None):
        """Checkpoint of the feedback state the decoding loop carries from step
        to step: the entropy history of the trigger (Section 3.2.1) and the EMA
        score table of the selection (Eq. 4-5), as host arrays.  `stream` is
        the stream the steps ran on (torch's current stream when None); it is
        synchronised first, so the checkpoint follows every queued step."""
        if self.d["hist"].is_cuda:
            (stream if stream is not None else torch.cuda.current_stream()).synchronize()
        return {k: self.d[k].cpu().numpy().copy() for k in self.STATE_KEYS}

    def load_state(self, state, stream=None):
        """Resume from a checkpoint taken by state() on a batch of the same
        shapes (history [B, l], counts [B], scores parallel to the tokens).

        The copies are ordered on `stream` -- the stream the steps run on
        (torch's current stream when None) -- behind any step still queued
        there, which reads and writes the same buffers; the call returns once
        the copies are done."""
        for k in self.STATE_KEYS:
            a = np.asarray(state[k])
            ref = self.host[k]
            if a.shape != ref.shape or a.dtype != ref.dtype:
                raise ValueError("VerifyStep.load_state: %s is %s %s, this batch needs %s %s"
                                 % (k, a.dtype, a.shape, ref.dtype, ref.shape))
        if not self.d["hist"].is_cuda:
            for k in self.STATE_KEYS:
                self.d[k].copy_(torch.from_numpy(np.ascontiguousarray(state[k])))
            return
        st = stream if stream is not None else torch.cuda.current_stream()
        with torch.cuda.stream(st):
            for k in self.STATE_KEYS:
                self.d[k].copy_(torch.from_numpy(np.ascontiguousarray(state[k])))
        st.synchronize()

    def save_state(self, path, stream=None):
        """state() written to an .npz file."""
        np.savez(path, **self.state(stream))

    def load_state_file(self, path, stream=None):
        with np.load(path) as f:
            self.load_state({k: f[k] for k in self.STATE_KEYS}, stream)


def arrays_from_workload(w):
    """Map a synthetic workload's fields onto the step's input names."""
    return dict(logits=w.logits, node_off=w.node_off, row_commit=w.row_commit, hist=w.hist,
                hist_n=w.hist_n, tokens=w.tokens, tok_off=w.tok_off, scores=w.scores, q=w.q, k=w.k,
                v=w.v, kv_off=w.kv_off, ctx_len=w.ctx_len, parents=w.parents,
                tree_tokens=w.tree_tokens, source=w.source, chain=w.chain, sel_pos=w.sel_pos)
