"""CPU-only checks of the C ABI: the library builds, loads and exports every
function include/heterofold.h declares, and host-side validation rejects bad
arguments before anything touches a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def B():
    from paper_2609_32259_gb300 import build, binding

    build.build()
    binding.lib()
    return binding


def declared_functions():
    text = open(os.path.join(ROOT, "include", "heterofold.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hf_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_binding_surface(B):
    assert declared_functions() == sorted(B.EXPORTED)


def test_library_exports_every_declared_symbol(B):
    L = B.lib()
    for name in declared_functions():
        assert hasattr(L, name), name
    out = os.popen(f"nm -D --defined-only {B.LIB_PATH}").read()
    exported = set(re.findall(r"\bT (hf_[a-z_0-9]+)\b", out))
    assert set(declared_functions()) <= exported


def test_status_strings(B):
    assert B.status_string(0) == "ok"
    assert B.status_string(1) == "invalid argument"
    assert B.status_string(99) == "unknown status"


def _desc(B, **over):
    kw = dict(L_s=4, H_s=2, D_s=64, L_r=6, H_r=4, D_r=32, dtype="bf16", layer_mode="paper3",
              align_mode="ta", s_tok_ptr=[0, 5], r_tok_ptr=[0, 6], d_row_ptr=16, d_col=32,
              d_w=48, d_W=64, d_b=80, r=np.ones((6, 2)), theta_r=1e4)
    kw.update(over)
    return B.Desc(**kw)


@pytest.mark.parametrize("over,status", [
    (dict(L_s=0), 1),                                  # shapes must be positive
    (dict(s_tok_ptr=[0, 0]), 1),                       # receiver tokens without sender tokens
    (dict(r_tok_ptr=[1, 6]), 1),                       # pointers start at 0
    (dict(r=np.zeros((6, 2))), 1),                     # r must be positive (Eq. 3)
    (dict(D_s=48), 2),                                 # d_S not a multiple of 64 (bf16)
    (dict(D_r=48, H_r=8), 2),                          # head width not a multiple of 32
    (dict(H_r=3, D_r=32), 2),                          # d_R not a multiple of 128
    (dict(paged=True, block_size=16, n_blocks=0), 1),  # paged layout incomplete
    (dict(d_W=None), 1),
    # optional fields
    (dict(layer_mode="explicit", seg_layer=np.zeros((6, 9, 1)), seg_w=1.0), 1),   # n_seg > 8
    (dict(layer_mode="explicit", seg_layer=np.zeros((6, 2, 3)), seg_w=1.0), 1),   # n_terms > 2
    (dict(layer_mode="explicit", seg_layer=np.full((6, 2, 1), 4), seg_w=1.0), 1),  # layer >= L_s
    (dict(layer_mode="explicit", seg_layer=np.zeros((6, 1, 2)), seg_w=np.nan), 1),
    (dict(layer_mode="explicit"), 1),                                             # no table
    (dict(sender_k_rotated=True), 1),                  # no theta_s and no sender table
    (dict(sender_k_rotated=True, theta_s=1e4, D_s=256, H_s=1), 2),  # head wider than a stage
    (dict(sender_k_rotated=True, theta_s=1e4, D_s=64, H_s=1), 2),   # d_S = 64: not whole stages
    (dict(inv_freq_r=np.full(16, np.inf)), 1),
    (dict(s_row0=[3], sender_rows=7), 1),             # span of 5 rows from row 3 > 7 rows
    (dict(s_row0=[-1], sender_rows=70), 1),
    (dict(sender_rows=4), 1),                         # fewer cache rows than sender tokens
    (dict(round_built_operands=2), 1),                # a flag: 0 or 1
])
def test_plan_create_rejects(B, over, status):
    d = _desc(B, **over)
    h = ctypes.c_void_p(0)
    st = B.lib().hf_plan_create(ctypes.byref(d.c), ctypes.c_void_p(256), 1 << 30, None,
                                ctypes.byref(h))
    assert st == status, B.lib().hf_last_error()
    assert h.value is None
    assert B.lib().hf_last_error()


def test_plan_create_checks_workspace(B):
    d = _desc(B)
    need = B.plan_workspace_size(d)
    assert need > 0
    h = ctypes.c_void_p(0)
    st = B.lib().hf_plan_create(ctypes.byref(d.c), ctypes.c_void_p(256), need - 1, None,
                                ctypes.byref(h))
    assert st == B.HF_ERR_WORKSPACE
    st = B.lib().hf_plan_create(ctypes.byref(d.c), ctypes.c_void_p(260), need, None,
                                ctypes.byref(h))
    assert st == B.HF_ERR_WORKSPACE  # not 256-byte aligned


def test_workspace_grows_with_tokens(B):
    a = B.plan_workspace_size(_desc(B, r_tok_ptr=[0, 6]))
    b = B.plan_workspace_size(_desc(B, r_tok_ptr=[0, 60000]))
    assert b - a >= 5 * 4 * (60000 - 6) - 4096


@pytest.mark.parametrize("args", [
    dict(n_req=0), dict(capacity=3), dict(mode=7), dict(ptr_start=1), dict(no_sender=True)])
def test_align_build_rejects(B, args):
    s_ptr = np.array([0, 4], np.int32)
    r_ptr = np.array([0, 6], np.int32)
    if args.get("ptr_start"):
        r_ptr = np.array([1, 6], np.int32)
    if args.get("no_sender"):
        s_ptr = np.array([0, 0], np.int32)
    n_req = args.get("n_req", 1)
    cap = args.get("capacity", 100)
    mode = args.get("mode", 0)
    st = B.lib().hf_align_build(mode, n_req, s_ptr.ctypes.data_as(B._i32p),
                                r_ptr.ctypes.data_as(B._i32p), 16, 32, 48, 64, 80, cap, 96, None)
    assert st == B.HF_ERR_INVALID_ARGUMENT


def test_transfer_rejects_null_plan(B):
    assert B.lib().hf_transfer(None, 16, 32, None) == B.HF_ERR_INVALID_ARGUMENT


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    import paper_2609_32259_gb300.binding as binding
    monkeypatch.setattr(binding, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(binding, "_LIB", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        binding.lib()


def test_optional_fields_validate(B):
    """The optional descriptor fields pass host validation when consistent
    (a failure after validation is a CUDA error on this device-less host, or
    success where a GPU is present)."""
    ok = [dict(layer_mode="explicit", seg_layer=np.zeros((6, 2, 2)), seg_w=0.5),
          dict(sender_k_rotated=True, theta_s=5e5, s_pos0=[3]),
          dict(sender_k_rotated=True, inv_freq_s=np.ones(32)),
          dict(inv_freq_r=np.linspace(1.0, 1e-3, 16), theta_r=0.0),
          dict(s_row0=[60], sender_rows=65)]
    for over in ok:
        d = _desc(B, **over)
        need = B.plan_workspace_size(d)
        h = ctypes.c_void_p(0)
        st = B.lib().hf_plan_create(ctypes.byref(d.c), ctypes.c_void_p(256), need, None,
                                    ctypes.byref(h))
        assert st in (B.HF_OK, B.HF_ERR_CUDA), (over, st, B.lib().hf_last_error())
        if st == B.HF_OK:
            B.lib().hf_plan_destroy(h)


def test_rotated_sender_workspace_holds_sender_positions(B):
    a = B.plan_workspace_size(_desc(B, s_tok_ptr=[0, 50000]))
    b = B.plan_workspace_size(_desc(B, s_tok_ptr=[0, 50000], sender_k_rotated=True, theta_s=1e4))
    assert b - a >= 4 * 50000 - 256


def test_debug_stalled_transfer_rejects_empty_plan(B):
    # the bounded-wait test hook validates on the host before any launch
    with pytest.raises(B.HFError) as e:
        B.debug_transfer_stalled(B.Plan(None, None, None), None, None)
    assert e.value.status == B.HF_ERR_INVALID_ARGUMENT
