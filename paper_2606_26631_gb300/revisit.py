"""A bundle of device buffers for repeated revisit calls.

``Revisit`` owns the outputs and the workspace of one batch shape and keeps
the descriptors, so a decode loop (or a benchmark) can call the library again
and again without rebuilding them. ``run_from_host`` is the end-to-end form:
it copies the step's selection, text positions and cache lengths from pinned
host memory, runs the call and reads the step's results back.
"""
from __future__ import annotations

from typing import Optional

import torch

from . import _binding as B


class Revisit:
    def __init__(self, cfg: B.RopeCfg, store_k, store_v, coords, cache_k, cache_v, block_table,
                 seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in, mode: int = B.MODE_PCR,
                 L: int = 2, flags: int = 0, want_pos: bool = True, want_slot: bool = True):
        dev = store_k.device
        self.cfg = cfg
        self.mode, self.L, self.flags = mode, L, flags
        self.store = B.store_desc(store_k, store_v, coords)
        if block_table is None:
            self.cache = B.cache_contiguous(cache_k, cache_v)
        else:
            self.cache = B.cache_paged(cache_k, cache_v, block_table)
        self.inputs = dict(seq_rev_off=seq_rev_off, rev_tok_off=rev_tok_off, idx=idx, p_txt=p_txt,
                           cache_len_in=cache_len_in, block_table=block_table)
        self.batch = B.revisit_batch(seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in)
        nB, K = self.batch.n_seqs, self.batch.total_k
        self.cache_len_out = torch.zeros(nB, dtype=torch.int32, device=dev)
        self.next_pos = torch.zeros(nB, dtype=torch.int64, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.pos = torch.zeros((K, 3), dtype=torch.float64, device=dev) if want_pos else None
        self.slot = torch.zeros(K, dtype=torch.int32, device=dev) if want_slot else None
        self.out = B.outputs(self.cache_len_out, self.next_pos, self.status, self.pos, self.slot)
        nbytes = B.workspace_size(K)
        self.workspace = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=dev)
        self._host = None

    def _args(self):
        return (self.cfg, self.store, self.cache, self.batch, self.out, self.mode, self.L,
                self.flags, self.workspace)

    def run(self, stream=None):
        """prcr_rebind_inject (plan kernel, then rebind + inject kernel)."""
        return B.rebind_inject(*self._args(), stream=stream)

    def run_plan(self, stream=None):
        return B.plan(*self._args(), stream=stream)

    def run_apply(self, stream=None):
        return B.rebind_apply(*self._args(), stream=stream)

    def status_value(self) -> int:
        return int(self.status.item()) & 0xFFFFFFFF

    # ------------------------------------------------------------------
    # end to end from host buffers
    # ------------------------------------------------------------------
    def host_inputs(self):
        """Pinned host copies of the per-step inputs (selection CSR, p_txt,
        cache lengths, block table) and of the per-step results."""
        if self._host is None:
            h = {k: v.cpu().pin_memory() for k, v in self.inputs.items() if v is not None}
            h["cache_len_out"] = torch.zeros_like(self.cache_len_out, device="cpu").pin_memory()
            h["next_pos"] = torch.zeros_like(self.next_pos, device="cpu").pin_memory()
            h["status"] = torch.zeros(1, dtype=torch.int32).pin_memory()
            self._host = h
        return self._host

    def h2d_bytes(self) -> int:
        h = self.host_inputs()
        return sum(h[k].numel() * h[k].element_size() for k in self.inputs if self.inputs[k] is not None)

    def d2h_bytes(self) -> int:
        h = self.host_inputs()
        return sum(h[k].numel() * h[k].element_size() for k in ("cache_len_out", "next_pos", "status"))

    def run_from_host(self, stream: Optional[torch.cuda.Stream] = None) -> int:
        """Copy this step's inputs host->device, run the call, copy the step's
        results (cache lengths, next positions, status) back and wait for
        them. Returns the status word."""
        h = self.host_inputs()
        s = stream or torch.cuda.current_stream()
        with torch.cuda.stream(s):
            for k, dv in self.inputs.items():
                if dv is not None:
                    dv.copy_(h[k], non_blocking=True)
            self.status.zero_()
            B.rebind_inject(*self._args(), stream=s)
            h["cache_len_out"].copy_(self.cache_len_out, non_blocking=True)
            h["next_pos"].copy_(self.next_pos, non_blocking=True)
            h["status"].copy_(self.status, non_blocking=True)
        s.synchronize()
        return int(h["status"].item()) & 0xFFFFFFFF
