"""One speculative step's attention through the C ABI (Algorithm 2: sparsify, Draft x gamma,
Verify), with preallocated outputs and workspace so the step can be captured in a CUDA graph."""

from __future__ import annotations

import torch

from . import binding as B


class SpecStep:
    """Runs bd_select_budget, gamma x bd_draft_attn and bd_verify_attn for one layer.

    The same object may serve many layers of one shape (the workspace is reused; calls
    on one stream are ordered)."""

    def __init__(self, batch, h_q, h_kv, head_dim, t_ctx, t_cap, budget, n_sink, n_recent,
                 window=32, gamma=5, chunk=1, device="cuda", seq_lens=None):
        """seq_lens: optional int32 device tensor [batch] of per-sequence context lengths
        (t_ctx is then the longest; bd_advance moves them on the device)."""
        self.seq_lens = seq_lens
        self.shape = B.make_shape(batch, h_q, h_kv, head_dim, t_ctx, t_cap, seq_lens)
        self.budget, self.n_sink, self.n_recent = budget, n_sink, n_recent
        self.window, self.gamma, self.chunk = window, gamma, chunk
        self.ws = B.Workspace.for_step(self.shape, budget, window, gamma, device)
        dev = torch.device(device)
        self.idx = torch.empty(batch, h_kv, budget, dtype=torch.int32, device=dev)
        self.count = torch.empty(batch, h_kv, dtype=torch.int32, device=dev)
        self.draft_o = torch.empty(gamma, batch, h_q, head_dim, dtype=torch.bfloat16, device=dev)
        self.draft_lse = torch.empty(gamma, batch, h_q, dtype=torch.float32, device=dev)
        self.verify_o = torch.empty(batch, h_q, gamma + 1, head_dim, dtype=torch.bfloat16, device=dev)
        self.verify_lse = torch.empty(batch, h_q, gamma + 1, dtype=torch.float32, device=dev)

    def bind_outputs(self, idx, count, draft_o, draft_lse, verify_o, verify_lse):
        """Directs the following calls' results into these tensors (same shapes and dtypes as
        the ones allocated here)."""
        self.idx, self.count = idx, count
        self.draft_o, self.draft_lse = draft_o, draft_lse
        self.verify_o, self.verify_lse = verify_o, verify_lse

    @classmethod
    def for_workload(cls, wl, budget=None, n_recent=None, chunk=1, device="cuda"):
        b = wl.budget if budget is None else budget
        r = wl.n_recent if n_recent is None else n_recent
        return cls(wl.batch, wl.h_q, wl.h_kv, wl.head_dim, wl.t_ctx, wl.t_cap, b, wl.n_sink, r,
                   wl.window, wl.gamma, chunk, device)

    def select(self, k_cache, q_win, window_lse=None, stream=None, window_ready=False):
        """window_ready: q_win, window_lse and the per-sequence lengths were not written by the
        kernel launched just before this call (BD_SELECT_WINDOW_READY), so they may be read
        while it finishes."""
        B.bd_select_budget(self.shape, k_cache, q_win, window_lse, self.window, self.budget, self.n_sink,
                           self.n_recent, self.chunk, self.idx, self.count, self.ws, stream,
                           flags=B.BD_SELECT_WINDOW_READY if window_ready else 0)

    def draft(self, j, q_j, k_cache, v_cache, stream=None, view_ready=False):
        """Draft pass j.  view_ready: the selection was not written by the kernel launched
        just before this one (true for every pass after the first of a step), so the pass may
        gather the view while that kernel finishes (BD_DRAFT_VIEW_READY)."""
        B.bd_draft_attn(self.shape, q_j, k_cache, v_cache, self.idx, self.count, self.budget, j,
                        self.draft_o[j], self.draft_lse[j], self.ws, stream,
                        flags=B.BD_DRAFT_VIEW_READY if view_ready else 0)

    def verify(self, q_verify, k_cache, v_cache, stream=None):
        B.bd_verify_attn(self.shape, q_verify, self.gamma + 1, k_cache, v_cache, self.verify_o,
                         self.verify_lse, self.ws, stream)

    def run(self, k_cache, v_cache, q_win, q_draft, q_verify, window_lse=None, stream=None):
        self.select(k_cache, q_win, window_lse, stream)
        for j in range(self.gamma):
            self.draft(j, q_draft[j], k_cache, v_cache, stream, view_ready=j > 0)
        self.verify(q_verify, k_cache, v_cache, stream)

    def window_lse(self, k_cache, q_win, out=None, stream=None):
        """LSE of the window queries over their causal prefixes, computed by the verify
        kernel (what a previous verify / prefill step leaves behind for carry mode).

        The window rows form a verify block that starts W positions before the context's
        end.  With per-sequence lengths, sequence b's rows sit at seq_lens[b] - W ..
        seq_lens[b] - 1, so every length must exceed the window W."""
        lens = None
        if self.seq_lens is not None:
            ts = torch.cuda.ExternalStream(stream) if isinstance(stream, int) else \
                (stream or torch.cuda.current_stream())
            with torch.cuda.stream(ts):
                lens = torch.sub(self.seq_lens, self.window)          # where each window block starts
            lens.record_stream(ts)
        sh = B.make_shape(self.shape.batch, self.shape.h_q, self.shape.h_kv, self.shape.head_dim,
                          self.shape.t_ctx - self.window, self.shape.t_cap, lens)
        if out is None:
            out = torch.empty(self.shape.batch, self.shape.h_q, self.window, dtype=torch.float32,
                              device=k_cache.device)
        ws = B.Workspace(B.bd_workspace_size(sh, B.BD_OP_VERIFY, 1, self.window), k_cache.device)
        B.bd_verify_attn(sh, q_win, self.window, k_cache, None, None, out, ws, stream)
        return out
