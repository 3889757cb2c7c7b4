"""Owner of the device buffers behind one wf_handle (marshalling only).

Uploads a synthetic parameter set as bf16 torch tensors, allocates the
workspace and the output buffers, and forwards every call to the C ABI in
`binding`.  No arithmetic of the method happens here.
"""
from __future__ import annotations

import numpy as np

from . import binding as B


def _bf16_tensor(bits, device):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device, non_blocking=False)


def upload_weights(ws, device="cuda") -> dict:
    """Device copies of a synthetic.WeightSet (bf16)."""
    up = lambda d: {k: _bf16_tensor(v, device) for k, v in d.items()}
    return {
        "target": up(ws.target),
        "target_layers": [up(lw) for lw in ws.target_layers],
        "drafter": up(ws.drafter),
        "drafter_layers": [up(lw) for lw in ws.drafter_layers],
    }


class Session:
    def __init__(self, cfg, weights, max_batch: int, max_ctx: int | None = None,
                 device="cuda", stream=None, keep_logits: bool = False):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.device = device
        self.max_batch = max_batch
        self.max_ctx = max_ctx or cfg.max_pos
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self.dev_weights = weights if isinstance(weights, dict) else upload_weights(weights, device)
        self.ccfg = B.make_config(cfg)
        self._structs = B.weight_structs(self.dev_weights, cfg.n_layers, cfg.n_draft_layers)
        self.ws_bytes = B.wf_workspace_bytes(self.ccfg, max_batch, self.max_ctx)
        self.workspace = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        tw, dw = self._structs[0], self._structs[1]
        self.h = B.wf_create(self.ccfg, tw, dw, max_batch, self.max_ctx, self.workspace,
                             self.ws_bytes, self.stream)
        if keep_logits:
            B.wf_set_option(self.h, B.WF_OPT_KEEP_LOGITS, 1)
        K = cfg.block_k
        self.out_tokens = torch.full((max_batch, K + 1), -1, dtype=torch.int32, device=device)
        self.out_count = torch.zeros(max_batch, dtype=torch.int32, device=device)

    def close(self):
        if self.h:
            B.wf_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _i32(self, a):
        return self.torch.as_tensor(np.ascontiguousarray(a, dtype=np.int32), device=self.device)

    # ----------------------------------------------------------- calls --
    def prefill(self, slots, enc_bits, prompt, budget, sp=None):
        """slots [n]; enc_bits uint16 [n, T, d] (bf16 bits) or a device bf16
        tensor; prompt int32 [n, P]; budget int32 [n].  Returns first tokens."""
        n, P = np.asarray(prompt).shape
        enc = enc_bits if not isinstance(enc_bits, np.ndarray) else _bf16_tensor(enc_bits, self.device)
        d_slots, d_prompt, d_budget = self._i32(slots), self._i32(prompt), self._i32(budget)
        first = self.torch.empty(n, dtype=self.torch.int32, device=self.device)
        B.wf_prefill_cross_kv(self.h, n, d_slots, enc, d_prompt, P, d_budget, first, sp,
                              self.stream)
        self._keep = (d_slots, d_prompt, d_budget, enc)
        return first

    def step(self, forced=None, sp=None, forced_q=None):
        """forced: proposals [max_batch, K]; forced_q: a device fp32 tensor
        [max_batch, K, vocab] of the logits they were drawn from (sampling)."""
        f = None if forced is None else (forced if not isinstance(forced, np.ndarray) else self._i32(forced))
        B.wf_step(self.h, sp, f, forced_q, self.out_tokens, self.out_count, self.stream)
        self._keep_forced = (f, forced_q)
        return self.out_tokens, self.out_count

    def draft(self, sp=None):
        B.wf_draft(self.h, sp, self.stream)

    def verify_accept(self, forced=None, sp=None, forced_q=None):
        f = None if forced is None else (forced if not isinstance(forced, np.ndarray) else self._i32(forced))
        B.wf_verify_accept(self.h, sp, f, forced_q, self.out_tokens, self.out_count, self.stream)
        self._keep_forced = (f, forced_q)
        return self.out_tokens, self.out_count

    def greedy_step(self, sp=None):
        B.wf_greedy_step(self.h, sp, self.out_tokens, self.out_count, self.stream)
        return self.out_tokens, self.out_count

    def compact(self) -> int:
        return B.wf_compact(self.h, self.stream)

    def reset_slots(self, slots):
        d = self._i32(slots)
        B.wf_reset_slots(self.h, len(slots), d, self.stream)
        self._keep_reset = d

    def state(self) -> dict:
        return B.wf_get_state(self.h, self.max_batch, self.stream)

    def error(self, clear=False) -> int:
        return B.wf_get_error(self.h, clear, self.stream)

    def launches(self) -> int:
        return B.wf_last_launch_count(self.h)

    def view(self, which, dtype, shape):
        """A torch view of an internal workspace buffer (see wf_debug_view)."""
        ptr, nbytes = B.wf_debug_view(self.h, which)
        base = self.workspace.data_ptr()
        off = ptr - base
        n = int(np.prod(shape)) * self.torch.empty((), dtype=dtype).element_size()
        assert 0 <= off and off + n <= self.ws_bytes and n <= nbytes
        return self.workspace[off:off + n].view(dtype).view(*shape)
