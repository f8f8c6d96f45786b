"""ctypes binding of the C ABI in include/heterofold.h.

Argument marshalling only: every step of the transfer runs in the CUDA
library.  Device pointers may be given as torch tensors (their data_ptr()) or
plain integers; host arrays as numpy arrays.  If libheterofold.so has not
been built, every call raises RuntimeError: there is no fallback path.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG_DIR, "libheterofold.so")

# enums of heterofold.h
HF_OK = 0
HF_ERR_INVALID_ARGUMENT = 1
HF_ERR_UNSUPPORTED = 2
HF_ERR_CUDA = 3
HF_ERR_DEVICE_CHECK = 5
HF_ERR_WORKSPACE = 6

ALIGN_MODES = {"ta": 0, "overlap_mean": 1, "same_index": 2}
LAYER_MODES = {"paper3": 0, "interp": 1, "explicit": 2}
DTYPES = {"bf16": 0, "f32": 1}

CHECK_BITS = {
    0x01: "HF_CHECK_BAD_OFFSETS", 0x02: "HF_CHECK_BAD_COLUMN", 0x04: "HF_CHECK_BAD_ROW",
    0x08: "HF_CHECK_BAD_BLOCK", 0x10: "HF_CHECK_CAPACITY", 0x20: "HF_CHECK_TIMEOUT",
    0x40: "HF_CHECK_INTERNAL", 0x80: "HF_CHECK_POOL_WINDOW",
}

EXPORTED = ("hf_align_build", "hf_plan_workspace_size", "hf_plan_create", "hf_transfer",
            "hf_plan_destroy", "hf_plan_device_status", "hf_plan_distinct_rows",
            "hf_status_string", "hf_last_error", "hf_transfer_noalloc", "hf_transfer_host",
            "hf_transfer_batch", "hf_fold", "hf_recolor_workspace_size", "hf_recolor_fit",
            "hf_debug_transfer_stalled", "hf_debug_matmul_workspace_size",
            "hf_debug_matmul_f32")

_p = ctypes.c_void_p
_i32p = ctypes.POINTER(ctypes.c_int32)
_f32p = ctypes.POINTER(ctypes.c_float)


class PlanDesc(ctypes.Structure):
    """Mirror of hf_plan_desc."""
    _fields_ = [
        ("L_s", ctypes.c_int32), ("H_s", ctypes.c_int32), ("D_s", ctypes.c_int32),
        ("L_r", ctypes.c_int32), ("H_r", ctypes.c_int32), ("D_r", ctypes.c_int32),
        ("dtype", ctypes.c_int), ("layer_mode", ctypes.c_int), ("align_mode", ctypes.c_int),
        ("n_req", ctypes.c_int32),
        ("s_tok_ptr", _i32p), ("r_tok_ptr", _i32p), ("r_pos0", _i32p),
        ("d_row_ptr", _p), ("d_col", _p), ("d_w", _p),
        ("d_W", _p), ("d_b", _p), ("h_r", _f32p),
        ("theta_r", ctypes.c_double),
        ("d_knorm_w", _p), ("knorm_eps", ctypes.c_float),
        ("paged", ctypes.c_int32), ("block_size", ctypes.c_int32),
        ("n_blocks", ctypes.c_int32), ("max_blocks_per_req", ctypes.c_int32),
        ("d_block_table", _p),
        ("h_inv_freq_r", _f32p),
        ("sender_k_rotated", ctypes.c_int32), ("theta_s", ctypes.c_double),
        ("h_inv_freq_s", _f32p), ("s_pos0", _i32p),
        ("s_row0", _i32p), ("sender_rows", ctypes.c_int64),
        ("n_seg", ctypes.c_int32), ("n_terms", ctypes.c_int32),
        ("h_seg_layer", _i32p), ("h_seg_w", _f32p),
        ("round_built_operands", ctypes.c_int32),
        ("pool_before_map", ctypes.c_int32),
    ]


class HFError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: status {status}: {msg}")
        self.status = status


_LIB: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it first "
                "(python -c 'import __graft_entry__ as g; g.build()'); there is no CPU fallback")
        L = ctypes.CDLL(LIB_PATH)
        L.hf_align_build.argtypes = [ctypes.c_int, ctypes.c_int32, _i32p, _i32p, _p, _p, _p, _p,
                                     _p, ctypes.c_int64, _p, _p]
        L.hf_plan_workspace_size.argtypes = [ctypes.POINTER(PlanDesc), ctypes.POINTER(ctypes.c_size_t)]
        L.hf_plan_create.argtypes = [ctypes.POINTER(PlanDesc), _p, ctypes.c_size_t, _p,
                                     ctypes.POINTER(ctypes.c_void_p)]
        L.hf_transfer.argtypes = [_p, _p, _p, _p]
        L.hf_debug_transfer_stalled.argtypes = [_p, _p, _p, _p]
        L.hf_debug_transfer_stalled.restype = ctypes.c_int
        L.hf_plan_destroy.argtypes = [_p]
        L.hf_plan_device_status.argtypes = [_p, _p, _i32p]
        L.hf_plan_distinct_rows.argtypes = [_p, _p, _i32p]
        L.hf_transfer_noalloc.argtypes = [ctypes.POINTER(PlanDesc), _p, _p, _p]
        L.hf_transfer_noalloc.restype = ctypes.c_int
        L.hf_transfer_host.argtypes = [_p, _p, _p, _p, _p, ctypes.c_int32, _p]
        L.hf_transfer_host.restype = ctypes.c_int
        L.hf_transfer_batch.argtypes = [_p, _p, _p, ctypes.c_int32, _p]
        L.hf_transfer_batch.restype = ctypes.c_int
        L.hf_fold.argtypes = [ctypes.c_int, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
                              ctypes.c_int32, _p, _p, _p, _p, _p, _p, _p]
        L.hf_fold.restype = ctypes.c_int
        L.hf_recolor_workspace_size.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                                ctypes.POINTER(ctypes.c_size_t)]
        L.hf_recolor_workspace_size.restype = ctypes.c_int
        L.hf_recolor_fit.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                     _p, _p, _p, ctypes.c_float, _p, _p, _f32p, _i32p, _p,
                                     ctypes.c_size_t, _p]
        L.hf_recolor_fit.restype = ctypes.c_int
        L.hf_debug_matmul_workspace_size.argtypes = [ctypes.c_int32, ctypes.c_int32,
                                                     ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]
        L.hf_debug_matmul_workspace_size.restype = ctypes.c_int
        L.hf_debug_matmul_f32.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                          ctypes.c_float, _p, ctypes.c_int64, ctypes.c_int64, _p,
                                          ctypes.c_int64, ctypes.c_int64, ctypes.c_float, _p,
                                          ctypes.c_int64, _p, ctypes.c_size_t, _i32p, _p]
        L.hf_debug_matmul_f32.restype = ctypes.c_int
        L.hf_status_string.argtypes = [ctypes.c_int]
        L.hf_status_string.restype = ctypes.c_char_p
        L.hf_last_error.argtypes = []
        L.hf_last_error.restype = ctypes.c_char_p
        for name in ("hf_align_build", "hf_plan_workspace_size", "hf_plan_create", "hf_transfer",
                     "hf_plan_destroy", "hf_plan_device_status", "hf_plan_distinct_rows"):
            getattr(L, name).restype = ctypes.c_int
        _LIB = L
    return _LIB


def _check(status: int, where: str) -> None:
    if status != HF_OK:
        raise HFError(status, where, lib().hf_last_error().decode(errors="replace"))


def _dptr(x) -> Optional[int]:
    """Device pointer of a torch tensor (or an int / None)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _stream(stream) -> Optional[int]:
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def _host_i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _as_i32p(a: np.ndarray):
    return a.ctypes.data_as(_i32p)


def _host_f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32).reshape(-1))


def _f32_or_null(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(_f32p)


def align_build(mode: str, s_tok_ptr, r_tok_ptr, d_s_end, d_r_end, d_row_ptr, d_col, d_w,
                nnz_capacity: int, d_info, stream=None) -> None:
    """hf_align_build.  Host token pointers (numpy), device arrays (torch)."""
    s = _host_i32(s_tok_ptr)
    r = _host_i32(r_tok_ptr)
    st = lib().hf_align_build(ALIGN_MODES[mode], len(r) - 1, _as_i32p(s), _as_i32p(r),
                              _dptr(d_s_end), _dptr(d_r_end), _dptr(d_row_ptr), _dptr(d_col),
                              _dptr(d_w), int(nnz_capacity), _dptr(d_info), _stream(stream))
    _check(st, "hf_align_build")


class Desc:
    """Builds an hf_plan_desc and keeps its host arrays alive."""

    def __init__(self, *, L_s, H_s, D_s, L_r, H_r, D_r, dtype, layer_mode, align_mode,
                 s_tok_ptr, r_tok_ptr, d_row_ptr, d_col, d_w, d_W, d_b, r, theta_r,
                 r_pos0=None, d_knorm_w=None, knorm_eps=1e-6, paged=False, block_size=16,
                 n_blocks=0, max_blocks_per_req=0, d_block_table=None, inv_freq_r=None,
                 sender_k_rotated=False, theta_s=0.0, inv_freq_s=None, s_pos0=None,
                 seg_layer=None, seg_w=None, s_row0=None, sender_rows=0,
                 round_built_operands=False, pool_before_map=False):
        self._s = _host_i32(s_tok_ptr)
        self._r = _host_i32(r_tok_ptr)
        self._pos0 = None if r_pos0 is None else _host_i32(r_pos0)
        self._spos0 = None if s_pos0 is None else _host_i32(s_pos0)
        self._srow0 = None if s_row0 is None else _host_i32(s_row0)
        self._hr = np.ascontiguousarray(np.asarray(r, dtype=np.float32).reshape(-1))
        self._ifr = None if inv_freq_r is None else _host_f32(inv_freq_r)
        self._ifs = None if inv_freq_s is None else _host_f32(inv_freq_s)
        n_seg = n_terms = 0
        self._segl = self._segw = None
        if seg_layer is not None:
            sl = np.ascontiguousarray(np.asarray(seg_layer, dtype=np.int32))
            if sl.ndim != 3:
                raise ValueError("seg_layer must be [L_r][n_seg][n_terms]")
            n_seg, n_terms = int(sl.shape[1]), int(sl.shape[2])
            self._segl = sl.reshape(-1)
            self._segw = _host_f32(np.broadcast_to(np.asarray(seg_w, dtype=np.float32), sl.shape))
        self.c = PlanDesc(
            L_s=L_s, H_s=H_s, D_s=D_s, L_r=L_r, H_r=H_r, D_r=D_r,
            dtype=DTYPES[dtype], layer_mode=LAYER_MODES[layer_mode],
            align_mode=ALIGN_MODES[align_mode], n_req=len(self._r) - 1,
            s_tok_ptr=_as_i32p(self._s), r_tok_ptr=_as_i32p(self._r),
            r_pos0=_as_i32p(self._pos0) if self._pos0 is not None else None,
            d_row_ptr=_dptr(d_row_ptr), d_col=_dptr(d_col), d_w=_dptr(d_w),
            d_W=_dptr(d_W), d_b=_dptr(d_b), h_r=self._hr.ctypes.data_as(_f32p),
            theta_r=float(theta_r), d_knorm_w=_dptr(d_knorm_w), knorm_eps=float(knorm_eps),
            paged=int(bool(paged)), block_size=int(block_size), n_blocks=int(n_blocks),
            max_blocks_per_req=int(max_blocks_per_req), d_block_table=_dptr(d_block_table),
            h_inv_freq_r=_f32_or_null(self._ifr), sender_k_rotated=int(bool(sender_k_rotated)),
            theta_s=float(theta_s), h_inv_freq_s=_f32_or_null(self._ifs),
            s_pos0=_as_i32p(self._spos0) if self._spos0 is not None else None,
            s_row0=_as_i32p(self._srow0) if self._srow0 is not None else None,
            sender_rows=int(sender_rows),
            n_seg=n_seg, n_terms=n_terms,
            h_seg_layer=_as_i32p(self._segl) if self._segl is not None else None,
            h_seg_w=_f32_or_null(self._segw),
            round_built_operands=int(round_built_operands),
            pool_before_map=int(pool_before_map))


def plan_workspace_size(desc: Desc) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().hf_plan_workspace_size(ctypes.byref(desc.c), ctypes.byref(n)),
           "hf_plan_workspace_size")
    return int(n.value)


class Plan:
    """An hf_plan handle; destroy() (or garbage collection) releases it."""

    def __init__(self, handle: int, desc: Desc, workspace):
        self.handle = handle
        self.desc = desc
        self.workspace = workspace

    def destroy(self) -> None:
        if self.handle:
            _check(lib().hf_plan_destroy(self.handle), "hf_plan_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def plan_create(desc: Desc, workspace, stream=None) -> Plan:
    h = ctypes.c_void_p(0)
    nbytes = int(workspace.numel() * workspace.element_size()) if hasattr(workspace, "numel") else 0
    _check(lib().hf_plan_create(ctypes.byref(desc.c), _dptr(workspace), nbytes, _stream(stream),
                                ctypes.byref(h)), "hf_plan_create")
    return Plan(h.value, desc, workspace)


def transfer(plan: Plan, sender_kv, receiver_kv, stream=None) -> None:
    _check(lib().hf_transfer(plan.handle, _dptr(sender_kv), _dptr(receiver_kv), _stream(stream)),
           "hf_transfer")


def debug_transfer_stalled(plan: Plan, sender_kv, receiver_kv, stream=None) -> None:
    """Test hook: a transfer launch whose first map atom never arrives (the
    bounded waits end it with HF_CHECK_TIMEOUT in the plan's status)."""
    _check(lib().hf_debug_transfer_stalled(plan.handle, _dptr(sender_kv), _dptr(receiver_kv),
                                           _stream(stream)), "hf_debug_transfer_stalled")


def transfer_host(plan: Plan, h_sender_kv, d_sender_kv, d_receiver_kv, h_receiver_kv,
                  n_groups: int = 0, stream=None) -> None:
    """hf_transfer_host: caches in page-locked host memory (torch tensors made
    with pin_memory=True), copies overlapped with the computation;
    h_receiver_kv None keeps the receiver cache on the device."""
    _check(lib().hf_transfer_host(plan.handle, _dptr(h_sender_kv), _dptr(d_sender_kv),
                                  _dptr(d_receiver_kv), _dptr(h_receiver_kv), int(n_groups),
                                  _stream(stream)), "hf_transfer_host")


def transfer_batch(plans, senders, receivers, stream=None) -> None:
    """hf_transfer_batch: direction i = (plans[i], senders[i], receivers[i])."""
    n = len(plans)
    hp = (ctypes.c_void_p * max(n, 1))(*[p.handle for p in plans])
    sp = (ctypes.c_void_p * max(n, 1))(*[_dptr(x) for x in senders])
    rp = (ctypes.c_void_p * max(n, 1))(*[_dptr(x) for x in receivers])
    _check(lib().hf_transfer_batch(hp, sp, rp, n, _stream(stream)), "hf_transfer_batch")


def fold(dtype: str, W, b, B, G, W_final, b_final, stream=None) -> None:
    """hf_fold (Eq. 9): W [n_maps, d_R, K], b [n_maps, d_R], B [n_maps, d_R, rank],
    G [n_maps, rank, d_R] (torch device tensors; W_final/b_final may alias)."""
    n_maps, d_R, K = (int(x) for x in W.shape)
    rank = int(B.shape[-1])
    _check(lib().hf_fold(DTYPES[dtype], n_maps, d_R, K, rank, _dptr(W), _dptr(b), _dptr(B),
                         _dptr(G), _dptr(W_final), _dptr(b_final), _stream(stream)), "hf_fold")


def recolor_workspace_size(N: int, d_S: int, d_R: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().hf_recolor_workspace_size(int(N), int(d_S), int(d_R), ctypes.byref(n)),
           "hf_recolor_workspace_size")
    return int(n.value)


def recolor_fit(dtype: str, X, Y, w, W_out, b_out, workspace, reg: float = 0.0,
                stream=None, return_iters: bool = False):
    """hf_recolor_fit (Eq. 3-5): X [N, d_S], Y [N, d_R], w [N] device tensors;
    writes W_out [d_R, d_S] (= A^T) and b_out [d_R]; returns r (and the three
    iteration counts with return_iters)."""
    N, d_S = (int(x) for x in X.shape)
    d_R = int(Y.shape[1])
    r = ctypes.c_float(0.0)
    its = (ctypes.c_int32 * 3)()
    nbytes = int(workspace.numel() * workspace.element_size())
    _check(lib().hf_recolor_fit(DTYPES[dtype], N, d_S, d_R, _dptr(X), _dptr(Y), _dptr(w),
                                float(reg), _dptr(W_out), _dptr(b_out), ctypes.byref(r),
                                its, _dptr(workspace), nbytes, _stream(stream)),
           "hf_recolor_fit")
    return (float(r.value), list(its)) if return_iters else float(r.value)


def transfer_noalloc(desc: Desc, sender_kv, receiver_kv, stream=None) -> None:
    """hf_transfer_noalloc: plan + transfer with the library's built-in
    metadata array (no workspace, no allocation)."""
    _check(lib().hf_transfer_noalloc(ctypes.byref(desc.c), _dptr(sender_kv), _dptr(receiver_kv),
                                     _stream(stream)), "hf_transfer_noalloc")


def plan_device_status(plan: Plan, stream=None) -> int:
    v = ctypes.c_int32(0)
    st = lib().hf_plan_device_status(plan.handle, _stream(stream), ctypes.byref(v))
    if st not in (HF_OK, HF_ERR_DEVICE_CHECK):
        _check(st, "hf_plan_device_status")
    return int(v.value)


def plan_distinct_rows(plan: Plan, stream=None) -> int:
    v = ctypes.c_int32(0)
    _check(lib().hf_plan_distinct_rows(plan.handle, _stream(stream), ctypes.byref(v)),
           "hf_plan_distinct_rows")
    return int(v.value)


def status_string(status: int) -> str:
    return lib().hf_status_string(int(status)).decode()


def decode_check_bits(bits: int):
    return [name for b, name in CHECK_BITS.items() if bits & b]


def debug_matmul_f32(A, a_strides, B, b_strides, C, M, N, K, alpha=1.0, beta=0.0,
                     stream=None) -> int:
    """Test hook: C = alpha op(A) op(B) + beta C through hf_debug_matmul_f32;
    a_strides = (a_i, a_k), b_strides = (b_k, b_j) in elements; returns the
    kernel's error word (0 = clean)."""
    import torch
    n = ctypes.c_size_t(0)
    _check(lib().hf_debug_matmul_workspace_size(int(M), int(N), int(K), ctypes.byref(n)),
           "hf_debug_matmul_workspace_size")
    ws = torch.empty(int(n.value), dtype=torch.uint8, device=C.device)
    err = np.zeros(1, np.int32)
    _check(lib().hf_debug_matmul_f32(int(M), int(N), int(K), float(alpha), _dptr(A),
                                     int(a_strides[0]), int(a_strides[1]), _dptr(B),
                                     int(b_strides[0]), int(b_strides[1]), float(beta), _dptr(C),
                                     int(C.stride(0)), _dptr(ws), int(n.value), _as_i32p(err),
                                     _stream(stream)), "hf_debug_matmul_f32")
    return int(err[0])
