"""Device-resident decode batch: uploads a workload's tensors and runs the
three C-ABI calls of one step (pad_plan -> pad_kv_append -> pad_event_decode_attn).

PyTorch is used only for device memory and streams; every step of the path
runs in libpad's kernels.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as B


def bits_to_bf16(a: np.ndarray, device) -> torch.Tensor:
    """uint16 bf16 bit patterns -> torch.bfloat16 tensor on ``device`` (exact)."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint16).view(np.int16))
    return t.view(torch.bfloat16).to(device)


class DeviceBatch:
    """All device state of one decode step for a ``synth.Workload``-like object."""

    def __init__(self, w, device="cuda", fill_nan: bool = True, flags: int = 0,
                 out_dtype: int = 0, num_sms: int = 0):
        self.w = w
        self.device = torch.device(device)
        self.problem = B.make_problem(w.h_q, w.h_kv, w.head_dim, w.page_size, w.scale,
                                      out_dtype=out_dtype, num_sms=num_sms, flags=flags)
        kp, vp = w.build_pools(fill_nan=fill_nan)
        self.k_pool = bits_to_bf16(kp, self.device)
        self.v_pool = bits_to_bf16(vp, self.device)
        self.k_prefix = bits_to_bf16(w.k_prefix, self.device)
        self.v_prefix = bits_to_bf16(w.v_prefix, self.device)
        # this step's inputs in one allocation (q | k_new | v_new) and its outputs in another
        # (out | lse), as a serving loop keeps them: the step executor then moves each group
        # with one copy
        qn, kn = w.q.size, w.k_new.size
        self.io_in = torch.empty(qn + 2 * kn, dtype=torch.bfloat16, device=self.device)
        self.q = self.io_in[:qn].view(w.q.shape)
        self.k_new = self.io_in[qn:qn + kn].view(w.k_new.shape)
        self.v_new = self.io_in[qn + kn:].view(w.v_new.shape)
        self.q.copy_(bits_to_bf16(w.q, self.device))
        self.k_new.copy_(bits_to_bf16(w.k_new, self.device))
        self.v_new.copy_(bits_to_bf16(w.v_new, self.device))
        self.page_table = torch.from_numpy(w.page_table.copy()).to(self.device)
        used = w.page_table[w.page_table >= 0]
        self.cache = B.CacheState(w.n_pages, used_pages=used)
        ws = B.pad_workspace_size(self.problem, w.prefix_len, w.event_video)
        if ws == 0:
            raise B.PadError(1, B.lib().pad_last_error().decode())
        self.workspace = torch.zeros(ws, dtype=torch.uint8, device=self.device)
        odt = torch.float32 if out_dtype == 0 else torch.bfloat16
        ob = w.n_events * w.h_q * w.head_dim * (4 if out_dtype == 0 else 2)
        lb = w.n_events * w.h_q * 4
        self.io_out = torch.empty(ob + lb, dtype=torch.uint8, device=self.device)
        self.out = self.io_out[:ob].view(odt).view(w.n_events, w.h_q, w.head_dim)
        self.lse = self.io_out[ob:].view(torch.float32).view(w.n_events, w.h_q)
        self.plan = None
        self.rope = None           # (positions [E] host int32, cos_sin device fp32 [P, D])
        self.self_g = None         # (K per video, G index per event) for the self G-token mask
        self.causal = False        # the causal-attention mask variant

    def set_rope(self, positions, table):
        """Rotate q and k_new at ``positions`` with the fp32 table ``table`` (numpy
        [max_position, D]) in every later step."""
        self.rope = (np.ascontiguousarray(positions, dtype=np.int32),
                     torch.from_numpy(np.ascontiguousarray(table, dtype=np.float32)).to(self.device))

    def plan_step(self, stream=None):
        w = self.w
        if self.plan is not None:
            self.plan.destroy()
        self.plan = B.pad_plan(self.problem, self.cache, w.prefix_len, w.event_video, w.event_len,
                               page_table=self.page_table, max_pages=w.max_pages,
                               workspace=self.workspace, prefix_offset=w.prefix_offset,
                               stream=stream)
        if self.rope is not None:
            self.plan.set_rope(self.rope[0], self.rope[1])
        if self.self_g is not None:
            self.plan.set_g_visibility(B.G_SELF, self.self_g[0], self.self_g[1])
        if self.causal:
            self.plan.set_branch_visibility(B.BRANCH_CAUSAL)
        return self.plan

    def run_step(self, stream=None, q=None, k_new=None, v_new=None, out=None, lse=None,
                 one_call=False):
        """plan + append + attention (two calls, or pad_decode_step with ``one_call``);
        returns the plan (its new pages stay allocated)."""
        plan = self.plan_step(stream)
        q = self.q if q is None else q
        k_new = self.k_new if k_new is None else k_new
        v_new = self.v_new if v_new is None else v_new
        out = self.out if out is None else out
        lse = self.lse if lse is None else lse
        if one_call:
            B.pad_decode_step(plan, q, k_new, v_new, self.k_prefix, self.v_prefix, self.k_pool,
                              self.v_pool, out, lse, stream)
        else:
            B.pad_kv_append(plan, k_new, v_new, self.k_pool, self.v_pool, stream)
            B.pad_event_decode_attn(plan, q, self.k_prefix, self.v_prefix, self.k_pool, self.v_pool,
                                    out, lse, stream)
        return plan

    def release_new_pages(self, plan=None):
        """Return the pages the last plan took (keeps repeated steps idempotent)."""
        (plan or self.plan).release_new_pages(self.cache)

    def gather_branch(self, e: int, n_tokens: int):
        """Read branch e's first n_tokens K/V rows back through the device page table."""
        pt = self.page_table[e].cpu().numpy()
        ps = self.w.page_size
        ks, vs = [], []
        for t in range(n_tokens):
            pg = int(pt[t // ps])
            ks.append(self.k_pool[pg, :, t % ps, :])
            vs.append(self.v_pool[pg, :, t % ps, :])
        return torch.stack(ks), torch.stack(vs)
