"""RelaySGD with the state in host memory, streamed through the GPU.

For state larger than the GPU, or owned by the host, ``HostRelayRun`` keeps
x, the two message buffers and the counters in pinned host memory, in the
device layout (``[rows][ld]``), and steps them with the library's host-state
calls (relay_step_host, relay_steps_host; include/relaysum.h).  The library
streams the coordinates through the GPU in chunks: copy-in, the fused kernel
at the chunk's absolute coordinate offset, copy-out, overlapped on its own
streams; the counters are stepped once per step.

Only the message rows a step reads cross the link inward: a message arriving
at a leaf is consumed by the leaf's rebuild in the step that forms it (a
leaf's only outgoing message excludes its only incoming one).  The same rows
come back -- the state the next step needs -- unless ``full_output`` is set,
which brings every row of m^t back, as relay_step writes it.  Without it,
messages() marks the rows the host does not receive as NaN.

``steps(k)`` runs k steps per chunk visit (relay_steps on each chunk), so
the state crosses the link once per k steps.

Every coordinate of the method evolves independently and the noise is keyed
by the absolute coordinate, so the result equals a run with the whole state
resident on the device, bit for bit.  The centres are regenerated in the
kernel (relay_set_objective_generated), so no device copy of mu is needed.
All arithmetic and every copy run in the library; this module allocates the
buffers and keeps the bookkeeping.
"""
from __future__ import annotations

import numpy as np

from . import _native as nat


class HostRelayRun:
    """One tree, n workers, d coordinates, state in pinned host memory."""

    def __init__(self, n: int, d: int, edges, chunk: int = 1 << 22, buffers: int = 3,
                 device="cuda", mode: int = 1, c0: int = 0, received_sums: bool = True,
                 full_output: bool = False):
        import torch
        if chunk % 32 or chunk <= 0:
            raise ValueError("chunk must be a positive multiple of 32")
        self.n, self.d, self.c0, self.mode = n, d, c0, mode
        self.device = torch.device(device)
        self.edges = np.asarray(edges, np.int32).reshape(-1, 2)
        self.received_sums = received_sums
        self.h = nat.relay_create(n, d, self.edges)
        nat.relay_set_received_sums(self.h, received_sums)
        nat.relay_set_rebuild_mode(self.h, mode)
        nat.relay_set_coord_offset(self.h, c0)
        self.E = nat.relay_num_edges(self.h)
        self.rows = nat.relay_message_rows(self.h)  # E, + the wide nodes' received sums
        self.ld = nat.relay_ld(self.h)
        self.chunk, self.buffers = chunk, buffers
        self.cw = min(chunk, max(32, (d + 31) // 32 * 32))
        self.nchunks = max(1, (d + self.cw - 1) // self.cw)
        # message rows a step reads: all but those arriving at a leaf (and
        # every received-sum row)
        if self.E > 0:
            _, _, node, pos = nat.relay_program(self.h)
            unread = {int(pos[node[i][1]][0]) for i in range(n) if node[i][0] == 1}
            self.kept_rows = [e for e in range(self.rows) if e not in unread]
        else:
            self.kept_rows = []
        pin = dict(dtype=torch.float32, pin_memory=True)
        ld1 = max(self.ld, 1)
        self.x_h = torch.zeros(n, ld1, **pin)
        self.msg_h = [torch.zeros(max(self.rows, 1), ld1, **pin) for _ in range(2)]
        self.counts_h = torch.zeros(max(self.E, 1), dtype=torch.int32, pin_memory=True)
        nbytes = nat.relay_host_staging_bytes(self.h, chunk, buffers)
        self.staging = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        self.plan = None
        self.set_full_output(full_output)
        self.t = 0
        self.cur = 0  # msg_h[cur] holds m^{t-1}

    def set_full_output(self, full_output: bool):
        """Whether a step copies every message row back (a new plan on the same staging)."""
        import torch
        self.full_output = bool(full_output)
        self.plan = None
        with torch.cuda.device(self.device):
            self.plan = nat.relay_host_plan_create(self.h, self.chunk, self.buffers, self.staging,
                                                   nat.RELAY_HOST_FULL_OUTPUT if full_output else 0)

    def init(self, x0_std: float, seed: int, mix, mu_scale: float, mu_seed: int, sigma: float):
        """x^0 (written chunk by chunk on the device, one shared Philox draw),
        zero messages and counters."""
        import torch
        mix = np.asarray(mix, dtype=np.float32)
        nat.relay_set_objective_generated(self.h, mix, mix.shape[1], mu_scale, mu_seed, sigma)
        for m in self.msg_h:
            m.zero_()
        self.counts_h.zero_()
        f32 = dict(dtype=torch.float32, device=self.device)
        xb = torch.empty(self.n, self.cw, **f32)
        mb = torch.empty(max(self.rows, 1), self.cw, **f32)
        cb = torch.empty(max(self.E, 1), dtype=torch.int32, device=self.device)
        for k in range(self.nchunks):
            lo = k * self.cw
            w = min(self.cw, self.d - lo)
            hc = nat.relay_create(self.n, w, self.edges)
            nat.relay_set_received_sums(hc, self.received_sums)
            nat.relay_set_strides(hc, self.cw, self.cw)
            nat.relay_set_coord_offset(hc, self.c0 + lo)
            with torch.cuda.device(self.device):
                nat.relay_init(hc, xb, mb, None, cb, x0_std, seed)
            wq = (w + 3) // 4 * 4
            self.x_h[:, lo:lo + wq].copy_(xb[:, :wq])
        torch.cuda.synchronize(self.device)
        self.t = 0
        self.cur = 0

    def _stream(self):
        import torch
        return torch.cuda.current_stream(self.device)

    def step(self, lr: float, seed: int):
        """Enqueues one RelaySGD step (asynchronous; call sync() to wait)."""
        import torch
        with torch.cuda.device(self.device):
            nat.relay_step_host(self.plan, self.x_h, self.msg_h[self.cur], self.msg_h[1 - self.cur], self.counts_h,
                                lr, seed, self.t, self._stream())
        self.cur = 1 - self.cur
        self.t += 1

    def steps(self, k: int, lr: float, seed: int):
        """Enqueues k steps with one relay_steps call per chunk visit, so the
        state crosses the host link once per k steps instead of once per
        step.  Afterwards the host holds x, the counters and m^{t+k-1} (the
        rows copied back), equal bit for bit to k step() calls; the other
        message buffer is not kept."""
        import torch
        k = int(k)
        if k <= 0:
            return
        dst = self.cur ^ (k & 1)
        with torch.cuda.device(self.device):
            nat.relay_steps_host(self.plan, self.x_h, self.msg_h[self.cur], self.msg_h[dst], self.counts_h, lr, seed,
                                 self.t, k, self._stream())
        self.cur = dst
        self.t += k

    def sync(self):
        import torch
        torch.cuda.synchronize(self.device)

    def bytes_per_step(self):
        """(host-to-device, device-to-host) bytes copied per step."""
        return nat.relay_host_bytes(self.plan)

    def models(self):
        """x as a host [n][d] array (a copy)."""
        return self.x_h[:, :self.d].clone()

    def messages(self):
        """m^{t-1} as a host [E][d] array (a copy); without full_output the
        rows the host does not receive (messages arriving at leaves, which no
        later step reads) are NaN."""
        import torch
        out = self.msg_h[self.cur][:self.E, :self.d].clone()
        if not self.full_output:
            dropped = [e for e in range(self.E) if e not in set(self.kept_rows)]
            if dropped:
                out[dropped] = torch.nan
        return out
