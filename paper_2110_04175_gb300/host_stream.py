"""RelaySGD with the state in host memory, streamed through the GPU.

For state larger than the GPU, or owned by the host, ``HostRelayRun`` keeps
x, the two message buffers and the counters in pinned host memory, laid out
in coordinate chunks (``[chunk][rows][cw]``, so each chunk of each array is
one contiguous block).  A step:

1. copies the counters in and runs the counter kernel once (Alg. 1 counters
   are per edge, not per coordinate);
2. streams the chunks through a ring of device buffers on three CUDA
   streams -- host-to-device copies, the fused kernel (relay_step_models on
   a handle whose coordinate offset is the chunk's absolute position), and
   device-to-host copies -- so both copy directions and the kernels overlap;
3. copies the counters out.

``steps(k)`` instead runs k steps per chunk visit (one relay_steps call per
chunk, the counters restored before each), so the state crosses the link
once per k steps.

Only the message rows that a later step reads cross the link.  A message
arriving at a leaf is consumed by the leaf's rebuild in the step that forms
it (a leaf's only outgoing message excludes its only incoming one), so those
rows are neither copied in nor copied out: the host keeps x, the counters
and every message row the next step reads, and messages() marks the rows it
does not keep as NaN.

Ordering: every reuse of a device buffer waits for the copy-out of the chunk
that last used it; a chunk's copy-in waits for the previous step's copy-out
of the same chunk (an event per chunk, as copies alternate between several
streams per direction); and the counters' copy-in waits for the last step's
copy-out.

Every coordinate of the method evolves independently and the noise is keyed
by the absolute coordinate, so the result equals a run with the whole state
resident on the device, bit for bit.  The centres are regenerated in the
kernel (relay_set_objective_generated), so no device copy of mu is needed.
All arithmetic runs in the library's kernels; this module only moves bytes
and orders the streams.
"""
from __future__ import annotations

import numpy as np

from . import _native as nat


class HostRelayRun:
    """One tree, n workers, d coordinates, state in pinned host memory."""

    def __init__(self, n: int, d: int, edges, chunk: int = 1 << 22, buffers: int = 3,
                 device="cuda", mode: int = 1, c0: int = 0, copy_streams: int = 2):
        import torch
        if chunk % 32 or chunk <= 0:
            raise ValueError("chunk must be a positive multiple of 32")
        self.n, self.d, self.c0, self.mode = n, d, c0, mode
        self.device = torch.device(device)
        self.cw = min(chunk, max(32, (d + 31) // 32 * 32))
        self.nchunks = max(1, (d + self.cw - 1) // self.cw)
        self.widths = [min(self.cw, d - k * self.cw) for k in range(self.nchunks)]
        # one handle per distinct chunk width; the offset is set per launch
        self.handles = {}
        for wdt in sorted(set(self.widths)):
            h = nat.relay_create(n, wdt, edges)
            nat.relay_set_rebuild_mode(h, mode)
            nat.relay_set_strides(h, self.cw, self.cw)
            self.handles[wdt] = h
        h0 = self.handles[self.widths[0]]
        self.E = nat.relay_num_edges(h0)
        E1 = max(self.E, 1)
        # message rows a later step reads: all but those arriving at a leaf,
        # as contiguous runs; only these cross the link, in both directions
        if self.E > 0:
            _, _, node, pos = nat.relay_program(h0)
            unread = {int(pos[node[i][1]][0]) for i in range(n) if node[i][0] == 1}
            self.kept_rows = [e for e in range(self.E) if e not in unread]
        else:
            self.kept_rows = []
        self.kept_runs = []
        for e in self.kept_rows:
            if self.kept_runs and self.kept_runs[-1][1] == e:
                self.kept_runs[-1][1] = e + 1
            else:
                self.kept_runs.append([e, e + 1])
        pin = dict(dtype=torch.float32, pin_memory=True)
        self.x_h = torch.empty(self.nchunks, n, self.cw, **pin)
        self.msg_h = [torch.empty(self.nchunks, E1, self.cw, **pin) for _ in range(2)]
        self.counts_h = torch.zeros(E1, dtype=torch.int32, pin_memory=True)
        f32 = dict(dtype=torch.float32, device=self.device)
        self.B = max(2, buffers, copy_streams)
        self.xb = [torch.empty(n, self.cw, **f32) for _ in range(self.B)]
        self.mib = [torch.empty(E1, self.cw, **f32) for _ in range(self.B)]
        self.mob = [torch.empty(E1, self.cw, **f32) for _ in range(self.B)]
        self.counts_d = torch.zeros(E1, dtype=torch.int32, device=self.device)
        # copies in each direction alternate between `copy_streams` streams so
        # that several copy engines can work at once
        self.s_ins = [torch.cuda.Stream(self.device) for _ in range(copy_streams)]
        self.s_outs = [torch.cuda.Stream(self.device) for _ in range(copy_streams)]
        self.s_in, self.s_out = self.s_ins[0], self.s_outs[0]
        self.s_comp = torch.cuda.Stream(self.device)
        self.in_done = [torch.cuda.Event() for _ in range(self.B)]
        self.comp_done = [torch.cuda.Event() for _ in range(self.B)]
        self.out_done = [torch.cuda.Event() for _ in range(self.B)]
        self.out_done_k = [torch.cuda.Event() for _ in range(self.nchunks)]  # chunk k written back
        self.counts_ready = torch.cuda.Event()  # counter kernel of this step done
        self.counts_saved = torch.cuda.Event()  # counters of the last step back on the host
        self.t = 0
        self.cur = 0  # msg_h[cur] holds m^{t-1}

    def _handle(self, k: int):
        h = self.handles[self.widths[k]]
        nat.relay_set_coord_offset(h, self.c0 + k * self.cw)
        return h

    def init(self, x0_std: float, seed: int, mix, mu_scale: float, mu_seed: int, sigma: float):
        """x^0, zero messages and counters, written chunk by chunk on the device."""
        import torch
        mix = np.asarray(mix, dtype=np.float32)
        for h in self.handles.values():
            nat.relay_set_objective_generated(h, mix, mix.shape[1], mu_scale, mu_seed, sigma)
        with torch.cuda.stream(self.s_comp):
            for k in range(self.nchunks):
                nat.relay_init(self._handle(k), self.xb[0], self.mib[0], None, self.counts_d,
                               x0_std, seed, self.s_comp)
                self.x_h[k].copy_(self.xb[0])
                self.msg_h[0][k].copy_(self.mib[0])
        self.counts_h.copy_(self.counts_d)
        torch.cuda.synchronize(self.device)
        self.t = 0
        self.cur = 0

    def step(self, lr: float, seed: int):
        """Enqueues one RelaySGD step (asynchronous; call sync() to wait)."""
        import torch
        src, dst = self.msg_h[self.cur], self.msg_h[1 - self.cur]
        with torch.cuda.stream(self.s_comp):
            # the last step's counters must be back on the host before they go in again
            self.s_comp.wait_event(self.counts_saved)
            self.counts_d.copy_(self.counts_h, non_blocking=True)
            nat.relay_step_counts(self.handles[self.widths[0]], self.counts_d, self.s_comp)
            self.counts_ready.record(self.s_comp)
        for k in range(self.nchunks):
            b = k % self.B
            s_in = self.s_ins[k % len(self.s_ins)]
            s_out = self.s_outs[k % len(self.s_outs)]
            with torch.cuda.stream(s_in):
                # the buffer's last chunk is out, and (through the same event on
                # in-order streams) so is this chunk's output of the last step
                s_in.wait_event(self.out_done[b])
                s_in.wait_event(self.out_done_k[k])
                self.xb[b].copy_(self.x_h[k], non_blocking=True)
                for lo, hi in self.kept_runs:
                    self.mib[b][lo:hi].copy_(src[k][lo:hi], non_blocking=True)
                self.in_done[b].record(s_in)
            self.s_comp.wait_event(self.in_done[b])
            nat.relay_step_models(self._handle(k), self.xb[b], self.mib[b], self.mob[b],
                                  self.counts_d, lr, seed, self.t, self.s_comp)
            self.comp_done[b].record(self.s_comp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(self.comp_done[b])
                self.x_h[k].copy_(self.xb[b], non_blocking=True)
                for lo, hi in self.kept_runs:
                    dst[k][lo:hi].copy_(self.mob[b][lo:hi], non_blocking=True)
                self.out_done[b].record(s_out)
                self.out_done_k[k].record(s_out)
        with torch.cuda.stream(self.s_out):
            self.s_out.wait_event(self.counts_ready)
            self.counts_h.copy_(self.counts_d, non_blocking=True)
            self.counts_saved.record(self.s_out)
        self.cur = 1 - self.cur
        self.t += 1

    def steps(self, k: int, lr: float, seed: int):
        """Enqueues k steps with one relay_steps call per chunk visit, so the
        state crosses the host link once per k steps instead of once per
        step.  The counters are per edge, not per coordinate: every chunk's
        call starts from the same c^{t-1}, restored from the host copy before
        it, and the last chunk's result goes back.  Afterwards the host holds
        x, the counters and m^{t+k-1} (the rows a later step reads), equal bit
        for bit to k step() calls; the other message buffer is not kept."""
        import torch
        k = int(k)
        if k <= 0:
            return
        src, dst = self.msg_h[self.cur], self.msg_h[self.cur ^ (k & 1)]
        with torch.cuda.stream(self.s_comp):
            self.s_comp.wait_event(self.counts_saved)
        for c in range(self.nchunks):
            b = c % self.B
            s_in = self.s_ins[c % len(self.s_ins)]
            s_out = self.s_outs[c % len(self.s_outs)]
            final = self.mob[b] if k & 1 else self.mib[b]  # the buffer step t+k-1 writes
            with torch.cuda.stream(s_in):
                s_in.wait_event(self.out_done[b])
                s_in.wait_event(self.out_done_k[c])
                self.xb[b].copy_(self.x_h[c], non_blocking=True)
                for lo, hi in self.kept_runs:
                    self.mib[b][lo:hi].copy_(src[c][lo:hi], non_blocking=True)
                self.in_done[b].record(s_in)
            with torch.cuda.stream(self.s_comp):
                self.s_comp.wait_event(self.in_done[b])
                self.counts_d.copy_(self.counts_h, non_blocking=True)
                nat.relay_steps(self._handle(c), self.xb[b], self.mib[b], self.mob[b], self.counts_d, lr, seed,
                                self.t, k, self.s_comp)
                self.comp_done[b].record(self.s_comp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(self.comp_done[b])
                self.x_h[c].copy_(self.xb[b], non_blocking=True)
                for lo, hi in self.kept_runs:
                    dst[c][lo:hi].copy_(final[lo:hi], non_blocking=True)
                self.out_done[b].record(s_out)
                self.out_done_k[c].record(s_out)
        with torch.cuda.stream(self.s_comp):
            self.counts_ready.record(self.s_comp)
        with torch.cuda.stream(self.s_out):
            self.s_out.wait_event(self.counts_ready)
            self.counts_h.copy_(self.counts_d, non_blocking=True)
            self.counts_saved.record(self.s_out)
        self.cur ^= k & 1
        self.t += k

    def sync(self):
        import torch
        torch.cuda.synchronize(self.device)

    def bytes_per_step(self):
        """(host-to-device, device-to-host) bytes copied per step."""
        rows = len(self.kept_rows)
        per_direction = (self.x_h.numel() + self.nchunks * rows * self.cw + self.counts_h.numel()) * 4
        return per_direction, per_direction

    def models(self):
        """x as a host [n][d] array (a copy)."""
        return self.x_h.permute(1, 0, 2).reshape(self.n, -1)[:, :self.d].clone()

    def messages(self):
        """m^{t-1} as a host [E][d] array (a copy); rows the host does not keep
        (messages arriving at leaves, which no later step reads) are NaN."""
        import torch
        m = self.msg_h[self.cur]
        out = m.permute(1, 0, 2).reshape(m.shape[1], -1)[:self.E, :self.d].clone()
        dropped = [e for e in range(self.E) if e not in set(self.kept_rows)]
        if dropped:
            out[dropped] = torch.nan
        return out
