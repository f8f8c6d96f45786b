"""One transfer direction end to end on one GPU: torch allocates the device
buffers, the C ABI does the work (alignment CSR, plan metadata, the fused
map).  No arithmetic of the method happens here.
"""

from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch

from . import binding as B


@dataclass
class PagedCache:
    block_table: np.ndarray  # [n_req, max_blocks] int32
    n_blocks: int
    block_size: int


class TransferJob:
    """Buffers and calls for one batch of requests.

    sender:   device tensor [L_s, 2, T_s, d_s] (bf16 or fp32)
    W:        device tensor [L_r, 2, d_r, K]  (A_final transposed)
    b:        device fp32 [L_r, 2, d_r];  r: host [L_r, 2]
    s_end / r_end: host int32 character-end offsets; s_tok_ptr / r_tok_ptr:
              host request pointers
    desc_options: the optional descriptor fields of binding.Desc
              (inv_freq_r, sender_k_rotated, theta_s, inv_freq_s, s_pos0,
              seg_layer, seg_w)
    """

    def __init__(self, *, L_s, H_s, D_s, L_r, H_r, D_r, dtype: str, align_mode: str,
                 layer_mode: str, s_tok_ptr, r_tok_ptr, s_end, r_end, sender, W, b, r,
                 theta_r: float, r_pos0=None, knorm_w=None, knorm_eps=1e-6,
                 paged: Optional[PagedCache] = None, device="cuda", receiver=None,
                 **desc_options):
        self.device = torch.device(device)
        self.s_tok_ptr = np.asarray(s_tok_ptr, np.int32)
        self.r_tok_ptr = np.asarray(r_tok_ptr, np.int32)
        self.T_s = int(self.s_tok_ptr[-1])
        self.T_r = int(self.r_tok_ptr[-1])
        self.align_mode = align_mode
        self.dtype = dtype
        self.L_r, self.H_r, self.D_r = L_r, H_r, D_r
        self.d_r = H_r * D_r
        self.paged = paged
        self.s_end = torch.as_tensor(np.asarray(s_end, np.int32)).to(self.device)
        self.r_end = torch.as_tensor(np.asarray(r_end, np.int32)).to(self.device)
        cap = self.T_r + (self.T_s if align_mode == "overlap_mean" else 0)
        self.nnz_capacity = max(cap, 1)
        self.row_ptr = torch.zeros(self.T_r + 1, dtype=torch.int32, device=self.device)
        self.col = torch.zeros(self.nnz_capacity, dtype=torch.int32, device=self.device)
        self.w = torch.zeros(self.nnz_capacity, dtype=torch.float32, device=self.device)
        self.info = torch.zeros(2, dtype=torch.int32, device=self.device)
        self.sender = sender
        self.W, self.b = W, b
        self.knorm_w = None if knorm_w is None else torch.as_tensor(knorm_w, dtype=torch.float32).to(self.device)
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        if receiver is not None:
            self.receiver = receiver
        elif paged is None:
            self.receiver = torch.empty((L_r, 2, self.T_r, self.d_r), dtype=tdt, device=self.device)
        else:
            self.receiver = torch.empty((L_r, 2, paged.n_blocks * paged.block_size, self.d_r),
                                        dtype=tdt, device=self.device)
        self.block_table = None
        if paged is not None:
            self.block_table = torch.as_tensor(np.ascontiguousarray(paged.block_table)).to(self.device)
        self.desc = B.Desc(
            L_s=L_s, H_s=H_s, D_s=D_s, L_r=L_r, H_r=H_r, D_r=D_r, dtype=dtype,
            layer_mode=layer_mode, align_mode=align_mode, s_tok_ptr=self.s_tok_ptr,
            r_tok_ptr=self.r_tok_ptr, d_row_ptr=self.row_ptr, d_col=self.col, d_w=self.w,
            d_W=W, d_b=b, r=r, theta_r=theta_r, r_pos0=r_pos0, d_knorm_w=self.knorm_w,
            knorm_eps=knorm_eps, paged=paged is not None,
            block_size=paged.block_size if paged else 16,
            n_blocks=paged.n_blocks if paged else 0,
            max_blocks_per_req=paged.block_table.shape[1] if paged else 0,
            d_block_table=self.block_table, **desc_options)
        ws = B.plan_workspace_size(self.desc)
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=self.device)
        self.plan: Optional[B.Plan] = None

    # -- the three calls of one transfer --------------------------------------
    def align(self, stream=None) -> None:
        B.align_build(self.align_mode, self.s_tok_ptr, self.r_tok_ptr, self.s_end, self.r_end,
                      self.row_ptr, self.col, self.w, self.nnz_capacity, self.info, stream)

    def make_plan(self, stream=None) -> B.Plan:
        if self.plan is not None:
            self.plan.destroy()
        self.plan = B.plan_create(self.desc, self.workspace, stream)
        return self.plan

    def transfer(self, stream=None, sender=None, receiver=None) -> None:
        B.transfer(self.plan, self.sender if sender is None else sender,
                   self.receiver if receiver is None else receiver, stream)

    def transfer_host(self, h_sender, h_receiver, n_groups=0, stream=None) -> None:
        """The transfer from/to page-locked host caches; self.sender and
        self.receiver serve as the device buffers."""
        B.transfer_host(self.plan, h_sender, self.sender, self.receiver, h_receiver, n_groups,
                        stream)

    def step(self, stream=None) -> None:
        """The whole hot path: alignment CSR, plan metadata, fused map."""
        self.align(stream)
        self.make_plan(stream)
        self.transfer(stream)

    # -- CUDA graphs ------------------------------------------------------------
    def capture(self) -> None:
        """Records one step as two CUDA graphs: ``prep`` (hf_align_build and
        hf_plan_create) and ``xfer`` (hf_transfer).  Every call of the step
        is stream-ordered and allocation-free, so the graphs replay the same
        kernels on the job's buffers: replays see the current contents of the
        sender cache, the offsets and the maps, and write the receiver cache
        and the plan workspace.  The plan created while recording is the
        job's plan afterwards (its host arrays went into the recorded kernel
        parameters)."""
        import torch
        self.step(torch.cuda.current_stream())  # kernel attributes, lazy module loading
        torch.cuda.synchronize()
        self.g_prep = torch.cuda.CUDAGraph()
        self.g_xfer = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.g_prep):
            s = torch.cuda.current_stream()
            self.align(s)
            self.make_plan(s)
        with torch.cuda.graph(self.g_xfer):
            self.transfer(torch.cuda.current_stream())

    def replay(self, prep: bool = True, xfer: bool = True) -> None:
        """Replays the recorded step on the current stream."""
        if prep:
            self.g_prep.replay()
        if xfer:
            self.g_xfer.replay()

    # -- inspection -------------------------------------------------------------
    def csr(self):
        nnz = int(self.info[0].item())
        return (self.row_ptr.cpu().numpy(), self.col[:nnz].cpu().numpy(),
                self.w[:nnz].cpu().numpy())

    def align_status(self) -> int:
        return int(self.info[1].item())

    def device_status(self, stream=None) -> int:
        return B.plan_device_status(self.plan, stream)

    def distinct_rows(self, stream=None) -> int:
        return B.plan_distinct_rows(self.plan, stream)

    def close(self) -> None:
        if self.plan is not None:
            self.plan.destroy()
            self.plan = None


def job_from_workload(w, tok, sender, W, b, r, *, paged=None, knorm_w=None, r_pos0=None,
                      device="cuda", receiver=None, **desc_options) -> TransferJob:
    """TransferJob for a workloads.Workload and its generated inputs; the
    workload's optional descriptor fields are passed on."""
    from . import workloads as W_
    opts = W_.desc_options(w, tok)
    opts.update(desc_options)
    pc = None
    if paged is not None:
        pc = PagedCache(paged.block_table, paged.n_blocks, w.block_size)
    return TransferJob(L_s=w.L_s, H_s=w.H_s, D_s=w.D_s, L_r=w.L_r, H_r=w.H_r, D_r=w.D_r,
                       dtype=w.dtype, align_mode=w.align_mode, layer_mode=w.layer_mode,
                       s_tok_ptr=tok.s_tok_ptr, r_tok_ptr=tok.r_tok_ptr, s_end=tok.s_end,
                       r_end=tok.r_end, sender=sender, W=W, b=b, r=r, theta_r=w.theta_r,
                       r_pos0=r_pos0, knorm_w=knorm_w, paged=pc, device=device,
                       receiver=receiver, **opts)
