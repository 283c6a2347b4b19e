"""Host-buffer driver of speculative steps: per-step inputs from pinned host memory, per-step
results back to pinned host memory, through the same C ABI calls as SpecStep.

Every step moves its inputs (window queries, drafter queries, the verify block, the
block's new K/V rows and the carried window LSE) host->device and its results (selection,
drafter and verifier outputs) device->host.  Queries and LSE are packed into one contiguous
buffer and the results into another (one copy each way per step instead of one per
tensor); the block's K/V rows go from pinned memory straight into the caches
(bd_write_block_rows).  Inputs and results move on two side streams, double-buffered:
step s+1's queries and step s-1's results move while step s's kernels run, and step s's
rows are written while its selection runs (the selection reads only the context rows).
The KV cache is model state that stays resident.
"""

from __future__ import annotations

import torch

from . import binding as B

_ALIGN = 256


class _Packed:
    """Named tensors laid out back to back (256-byte aligned) in one byte buffer."""

    def __init__(self, specs):
        self.specs = []          # (name, shape, dtype, offset, nbytes)
        off = 0
        for name, shape, dtype in specs:
            n = 1
            for s in shape:
                n *= s
            nbytes = n * torch.empty((), dtype=dtype).element_size()
            self.specs.append((name, tuple(shape), dtype, off, nbytes))
            off += (nbytes + _ALIGN - 1) // _ALIGN * _ALIGN
        self.nbytes = max(off, _ALIGN)

    def views(self, buf):
        return {name: buf[off: off + nb].view(dtype).view(shape) for name, shape, dtype, off, nb in self.specs}


class HostStepIO:
    """Runs speculative steps of one or more layers from host buffers.

    layers: list of (SpecStep, k_cache, v_cache, carry) per layer; carry=True if the
    layer's selection takes a carried window LSE (one more host input).  Inputs for step
    s are read from ``host_inputs(s % 2)`` and results land in ``host_outputs(s % 2)``;
    the buffers of a slot may be refilled / read once ``run`` has returned and the
    current stream has been synchronised.
    """

    def __init__(self, layers, device="cuda"):
        self.layers = layers
        specs_in, specs_out, specs_rows = [], [], []
        for l, (st, k_cache, _, carry) in enumerate(layers):
            sh = st.shape
            b, hq, hkv, d, g = sh.batch, sh.h_q, sh.h_kv, sh.head_dim, st.gamma
            bf = torch.bfloat16
            specs_in += [(f"q_win{l}", (b, hq, st.window, d), bf), (f"q_draft{l}", (g, b, hq, d), bf),
                         (f"q_verify{l}", (b, hq, g + 1, d), bf)]
            specs_rows.append((f"k_rows{l}", (b, hkv, g + 1, d), bf))
            specs_rows.append((f"v_rows{l}", (b, hkv, g + 1, d), bf))
            if carry:
                specs_in.append((f"lse{l}", (b, hq, st.window), torch.float32))
            specs_out += [(f"idx{l}", tuple(st.idx.shape), torch.int32), (f"count{l}", tuple(st.count.shape), torch.int32),
                          (f"draft_o{l}", tuple(st.draft_o.shape), bf),
                          (f"draft_lse{l}", tuple(st.draft_lse.shape), torch.float32),
                          (f"verify_o{l}", tuple(st.verify_o.shape), bf),
                          (f"verify_lse{l}", tuple(st.verify_lse.shape), torch.float32)]
        self.pin = _Packed(specs_in)
        self.prow = _Packed(specs_rows)
        self.pout = _Packed(specs_out)
        dev = torch.device(device)
        u8 = torch.uint8
        self.h_in = [torch.zeros(self.pin.nbytes, dtype=u8, pin_memory=True) for _ in range(2)]
        self.h_rows = [torch.zeros(self.prow.nbytes, dtype=u8, pin_memory=True) for _ in range(2)]
        self.d_in = [torch.zeros(self.pin.nbytes, dtype=u8, device=dev) for _ in range(2)]
        self.h_out = [torch.zeros(self.pout.nbytes, dtype=u8, pin_memory=True) for _ in range(2)]
        self.d_out = [torch.zeros(self.pout.nbytes, dtype=u8, device=dev) for _ in range(2)]
        self.in_stream = torch.cuda.Stream(device=dev)
        self.out_stream = torch.cuda.Stream(device=dev)

    @property
    def bytes_in(self):
        return sum(nb for *_, nb in self.pin.specs) + sum(nb for *_, nb in self.prow.specs)

    @property
    def bytes_out(self):
        return sum(nb for *_, nb in self.pout.specs)

    def host_inputs(self, slot):
        v = self.pin.views(self.h_in[slot])
        v.update(self.prow.views(self.h_rows[slot]))
        return v

    def host_outputs(self, slot):
        return self.pout.views(self.h_out[slot])

    def _bind(self, l, vout):
        self.layers[l][0].bind_outputs(vout[f"idx{l}"], vout[f"count{l}"], vout[f"draft_o{l}"],
                                       vout[f"draft_lse{l}"], vout[f"verify_o{l}"], vout[f"verify_lse{l}"])

    def run(self, n_steps):
        """Issues n_steps pipelined steps on the current stream (capturable in a CUDA graph).

        Step s+1's packed queries are copied during step s, once step s-1's kernels (the
        slot's last readers) are done; step s+1's K/V rows once step s's kernels are done;
        step s's results once its kernels are done.  Every wait of the compute stream on
        a copy sits just before a step's first draft pass, so the selection and verify
        kernels keep their programmatic (overlapping) launches: before step s's first draft
        pass it waits for its rows, for step s+1's queries and for step s-1's result copy
        (the last reader of the slot step s+1 writes)."""
        if n_steps < 1:
            return
        cs = torch.cuda.current_stream()
        xi, xo = self.in_stream, self.out_stream
        xi.wait_stream(cs)
        xo.wait_stream(cs)
        L = range(len(self.layers))
        g = self.layers[0][0].gamma

        def copy_queries(step):
            e = torch.cuda.Event()
            with torch.cuda.stream(xi):
                self.d_in[step % 2].copy_(self.h_in[step % 2], non_blocking=True)
                e.record(xi)
            return e

        def copy_rows(step):
            e = torch.cuda.Event()
            with torch.cuda.stream(xi):
                hr = self.prow.views(self.h_rows[step % 2])
                for l in L:
                    st, k_cache, v_cache, _ = self.layers[l]
                    B.bd_write_block_rows(st.shape, st.gamma + 1, hr[f"k_rows{l}"], hr[f"v_rows{l}"], k_cache,
                                          v_cache, xi)
                e.record(xi)
            return e

        q_ready = copy_queries(0)
        rows_ready = copy_rows(0)
        cs.wait_event(q_ready)
        done = [None] * n_steps
        drained = [None] * n_steps
        for s in range(n_steps):
            slot = s % 2
            if s + 1 < n_steps:
                if s >= 1:
                    xi.wait_event(done[s - 1])
                q_next = copy_queries(s + 1)
            vin = self.pin.views(self.d_in[slot])
            vout = self.pout.views(self.d_out[slot])
            for l in L:
                st, k_cache, _, carry = self.layers[l]
                self._bind(l, vout)
                # the slot's queries landed before the previous step's first draft pass
                st.select(k_cache, vin[f"q_win{l}"], vin[f"lse{l}"] if carry else None, window_ready=True)
            cs.wait_event(rows_ready)
            if s + 1 < n_steps:
                cs.wait_event(q_next)
            if s >= 1:
                cs.wait_event(drained[s - 1])
            for j in range(g):
                for l in L:
                    st, k_cache, v_cache, _ = self.layers[l]
                    self._bind(l, vout)
                    st.draft(j, vin[f"q_draft{l}"][j], k_cache, v_cache, view_ready=j > 0 or len(self.layers) > 1)
            for l in L:
                st, k_cache, v_cache, _ = self.layers[l]
                self._bind(l, vout)
                st.verify(vin[f"q_verify{l}"], k_cache, v_cache)
            done[s] = torch.cuda.Event()
            done[s].record(cs)
            if s + 1 < n_steps:
                xi.wait_event(done[s])
                rows_ready = copy_rows(s + 1)
            with torch.cuda.stream(xo):
                xo.wait_event(done[s])
                self.h_out[slot].copy_(self.d_out[slot], non_blocking=True)
                drained[s] = torch.cuda.Event()
                drained[s].record(xo)
        cs.wait_stream(xi)
        cs.wait_stream(xo)
