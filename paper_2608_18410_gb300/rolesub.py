"""Thin Python binding of librolesub.so (include/rolesub.h).

Argument marshalling only: every step of the hot path runs in the CUDA
library. torch provides device memory and streams. The functions named like
the C entry points take torch tensors (or raw integers for pointers) and
return nothing but raise RoleSubError on a non-OK status.

If the library is missing the import of this module fails loudly; there is
no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "librolesub.so")

F32, BF16 = 0, 1
VIS, LANG, PROP, ACT = 0, 1, 2, 3
NUM_KINDS = 4
PLAN_MAGIC = 0x42555352

STATUS = {0: "ROLESUB_OK", 1: "ROLESUB_EINVAL", 2: "ROLESUB_EUNSUPPORTED", 3: "ROLESUB_ECUDA",
          4: "ROLESUB_EDEVICE", 5: "ROLESUB_ETIMEOUT", 6: "ROLESUB_ETOOLARGE"}

# every symbol include/rolesub.h declares
EXPORTS = ("rolesub_plan_size", "rolesub_layout_plan", "rolesub_workspace_size",
           "rolesub_compress", "rolesub_attend", "rolesub_get_device_status",
           "rolesub_reset_device_status", "rolesub_status_string", "rolesub_version",
           "rolesub_launch_count", "rolesub_compress_static", "rolesub_compress_additive",
           "rolesub_budget_workspace_size", "rolesub_compress_budget", "rolesub_attend_budget",
           "rolesub_select_count", "rolesub_select_tokens", "rolesub_dense_workspace_size",
           "rolesub_compress_dense", "rolesub_attend_dense", "rolesub_static_device_status",
           "rolesub_static_scratch_bytes", "rolesub_wait_selftest")


class RoleSubError(RuntimeError):
    def __init__(self, fn, code):
        self.code = code
        super().__init__(f"{fn} failed: {STATUS.get(code, code)}")


class Shape(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("num_groups", ctypes.c_int32),
                ("role_dim", ctypes.c_int32), ("router_hidden", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class Segment(ctypes.Structure):
    _fields_ = [("episode", ctypes.c_int32), ("kind", ctypes.c_int32),
                ("n_tokens", ctypes.c_int32), ("k", ctypes.c_int32),
                ("token_row", ctypes.c_int64), ("packed_off", ctypes.c_int64),
                ("idx_off", ctypes.c_int64)]


class Episode(ctypes.Structure):
    _fields_ = [("row_begin", ctypes.c_int64), ("q_row_begin", ctypes.c_int64),
                ("n_cache", ctypes.c_int32), ("n_query", ctypes.c_int32),
                ("seg_begin", ctypes.c_int32), ("n_lang", ctypes.c_int32),
                ("lang_row_begin", ctypes.c_int64)]


class PlanHeader(ctypes.Structure):
    _fields_ = [("magic", ctypes.c_uint32), ("version", ctypes.c_uint32),
                ("num_episodes", ctypes.c_int32), ("num_segments", ctypes.c_int32),
                ("rows_per_layer", ctypes.c_int64), ("q_rows_per_layer", ctypes.c_int64),
                ("packed_elems_per_layer", ctypes.c_int64), ("idx_bytes_per_layer", ctypes.c_int64),
                ("routed_rows_per_layer", ctypes.c_int64), ("stored_rows_per_layer", ctypes.c_int64),
                ("max_cache_tokens", ctypes.c_int32), ("max_query_tokens", ctypes.c_int32),
                ("num_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("num_groups", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("off_segments", ctypes.c_int64), ("off_episodes", ctypes.c_int64),
                ("off_row_seg", ctypes.c_int64), ("off_routed_rows", ctypes.c_int64),
                ("off_stored_rows", ctypes.c_int64), ("total_bytes", ctypes.c_int64),
                ("num_route_tiles", ctypes.c_int32), ("reserved2", ctypes.c_int32),
                ("off_route_tiles", ctypes.c_int64)]


_vp = ctypes.c_void_p
_i32p = ctypes.POINTER(ctypes.c_int32)
_szp = ctypes.POINTER(ctypes.c_size_t)
_lib = None


def lib():
    """The loaded CUDA library; raises if it was not built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"librolesub.so not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        sp = ctypes.POINTER(Shape)
        L.rolesub_plan_size.argtypes = [ctypes.c_int32, _i32p, _szp]
        L.rolesub_layout_plan.argtypes = [sp, ctypes.c_int32, _i32p, _i32p, _i32p, _vp, ctypes.c_size_t]
        L.rolesub_workspace_size.argtypes = [sp, _vp, _szp]
        L.rolesub_compress.argtypes = ([sp, _vp, _vp] + [_vp] * 9 + [ctypes.c_float, ctypes.c_float]
                                       + [_vp, _vp, _vp, ctypes.c_size_t, _vp])
        L.rolesub_attend.argtypes = ([sp, _vp, _vp, _vp] + [ctypes.c_int64] * 3 + [_vp]
                                     + [ctypes.c_int64] * 3 + [_vp, _vp, _vp, ctypes.c_float, _vp,
                                                               _vp, ctypes.c_size_t, _vp])
        L.rolesub_get_device_status.argtypes = [_vp, _vp, _i32p, _i32p]
        L.rolesub_reset_device_status.argtypes = [_vp, _vp]
        L.rolesub_status_string.argtypes = [ctypes.c_int]
        L.rolesub_status_string.restype = ctypes.c_char_p
        L.rolesub_version.argtypes = []
        L.rolesub_version.restype = ctypes.c_int32
        L.rolesub_compress_static.argtypes = ([sp, _vp, _vp] + [_vp] * 9 + [ctypes.c_float, ctypes.c_float]
                                              + [_vp, _vp, _vp])
        L.rolesub_compress_additive.argtypes = ([sp, _vp, _vp] + [_vp] * 10 + [ctypes.c_float, ctypes.c_float]
                                                + [_vp, _vp, _vp, ctypes.c_size_t, _vp])
        L.rolesub_budget_workspace_size.argtypes = [sp, _vp, _szp]
        L.rolesub_compress_budget.argtypes = ([sp, _vp, _vp] + [_vp] * 11 + [ctypes.c_float, ctypes.c_float]
                                              + [_vp, _vp, _vp, _vp, ctypes.c_size_t, _vp])
        L.rolesub_attend_budget.argtypes = ([sp, _vp, _vp, _vp] + [ctypes.c_int64] * 3 + [_vp]
                                            + [ctypes.c_int64] * 3 + [_vp, _vp, _vp, _vp, ctypes.c_float, _vp,
                                                                      _vp, ctypes.c_size_t, _vp])
        L.rolesub_select_count.argtypes = [ctypes.c_int32, ctypes.c_double]
        L.rolesub_select_count.restype = ctypes.c_int32
        L.rolesub_select_tokens.argtypes = ([ctypes.c_int32] * 3 + [ctypes.c_double, _vp, _vp, ctypes.c_int32,
                                                                   ctypes.c_int32, _vp, _vp, _vp])
        L.rolesub_dense_workspace_size.argtypes = [sp, _vp, _szp]
        L.rolesub_compress_dense.argtypes = ([sp, _vp, _vp] + [_vp] * 9 + [ctypes.c_float, ctypes.c_float]
                                             + [_vp, _vp, _vp, ctypes.c_size_t, _vp])
        L.rolesub_attend_dense.argtypes = ([sp, _vp, _vp, _vp] + [ctypes.c_int64] * 3 + [_vp]
                                           + [ctypes.c_int64] * 3 + [_vp, _vp, _vp, ctypes.c_float, _vp,
                                                                     _vp, ctypes.c_size_t, _vp])
        L.rolesub_launch_count.argtypes = []
        L.rolesub_launch_count.restype = ctypes.c_uint64
        L.rolesub_static_device_status.argtypes = [_vp, _i32p, _i32p]
        L.rolesub_wait_selftest.argtypes = [ctypes.c_int64, _vp, _vp, _vp]
        L.rolesub_static_scratch_bytes.argtypes = []
        L.rolesub_static_scratch_bytes.restype = ctypes.c_size_t
        for name in EXPORTS:
            if name not in ("rolesub_status_string", "rolesub_version", "rolesub_launch_count",
                            "rolesub_select_count", "rolesub_static_scratch_bytes"):
                getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


def _check(fn, code):
    if code != 0:
        raise RoleSubError(fn, code)


def _ptr(x):
    """Device/host address of a tensor, an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_shape(L, H, dh, G, C, F, dtype):
    return Shape(L, H, dh, G, C, F, BF16 if dtype in ("bf16", BF16) else F32, 0)


def _aligned_buffer(nbytes, align=64):
    raw = np.zeros(nbytes + align, np.uint8)
    off = (-raw.ctypes.data) % align
    return raw[off:off + nbytes]


class Plan:
    """Host plan blob produced by rolesub_layout_plan, plus parsed views."""

    def __init__(self, shape: Shape, n_tok, k, n_query):
        n_tok = np.ascontiguousarray(n_tok, np.int32).reshape(-1)
        k = np.ascontiguousarray(k, np.int32).reshape(-1)
        n_query = np.ascontiguousarray(n_query, np.int32).reshape(-1)
        E = n_query.shape[0]
        sz = ctypes.c_size_t(0)
        _check("rolesub_plan_size", lib().rolesub_plan_size(E, n_tok.ctypes.data_as(_i32p), ctypes.byref(sz)))
        self.host = _aligned_buffer(max(int(sz.value), 16))
        _check("rolesub_layout_plan", lib().rolesub_layout_plan(
            ctypes.byref(shape), E, n_tok.ctypes.data_as(_i32p), k.ctypes.data_as(_i32p),
            n_query.ctypes.data_as(_i32p), self.host.ctypes.data, self.host.nbytes))
        self.shape = shape
        self.hdr = PlanHeader.from_buffer_copy(self.host[:ctypes.sizeof(PlanHeader)].tobytes())
        h = self.hdr
        self.segments = (Segment * h.num_segments).from_buffer_copy(
            self.host[h.off_segments:h.off_segments + ctypes.sizeof(Segment) * h.num_segments].tobytes()) \
            if h.num_segments else []
        self.episodes = (Episode * h.num_episodes).from_buffer_copy(
            self.host[h.off_episodes:h.off_episodes + ctypes.sizeof(Episode) * h.num_episodes].tobytes()) \
            if h.num_episodes else []
        self.dev = None

    @property
    def host_ptr(self):
        return self.host.ctypes.data

    def to_device(self, device="cuda"):
        import torch
        self.dev = torch.from_numpy(self.host[: self.hdr.total_bytes].copy()).to(device)
        return self.dev

    def budget_workspace_size(self):
        sz = ctypes.c_size_t(0)
        _check("rolesub_budget_workspace_size", lib().rolesub_budget_workspace_size(
            ctypes.byref(self.shape), self.host_ptr, ctypes.byref(sz)))
        return int(sz.value)

    def dense_workspace_size(self):
        sz = ctypes.c_size_t(0)
        _check("rolesub_dense_workspace_size", lib().rolesub_dense_workspace_size(
            ctypes.byref(self.shape), self.host_ptr, ctypes.byref(sz)))
        return int(sz.value)

    def workspace_size(self):
        sz = ctypes.c_size_t(0)
        _check("rolesub_workspace_size", lib().rolesub_workspace_size(
            ctypes.byref(self.shape), self.host_ptr, ctypes.byref(sz)))
        return int(sz.value)


# ---------------------------------------------------------------------------
# Entry points with the C names
# ---------------------------------------------------------------------------

def rolesub_compress(shape, plan: Plan, plan_dev, h, v, R, W_re, b_re, W1, b1, W2, b2, alpha_role,
                     alpha_lang, packed_v, idx, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_compress", lib().rolesub_compress(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(h), _ptr(v), _ptr(R), _ptr(W_re),
        _ptr(b_re), _ptr(W1), _ptr(b1), _ptr(W2), _ptr(b2), float(alpha_role), float(alpha_lang),
        _ptr(packed_v), _ptr(idx), _ptr(workspace), int(ws_bytes), _stream(stream)))


def rolesub_compress_additive(shape, plan: Plan, plan_dev, h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l,
                              alpha_role, alpha_lang, packed_v, idx, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_compress_additive", lib().rolesub_compress_additive(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(h), _ptr(v), _ptr(R), _ptr(W_re),
        _ptr(b_re), _ptr(W_v), _ptr(b_v), _ptr(W_role), _ptr(W_l), _ptr(b_l), float(alpha_role),
        float(alpha_lang), _ptr(packed_v), _ptr(idx), _ptr(workspace), int(ws_bytes), _stream(stream)))


def rolesub_compress_budget(shape, plan: Plan, plan_dev, h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l, u,
                            alpha_role, alpha_lang, packed_v, idx, k_tok, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_compress_budget", lib().rolesub_compress_budget(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(h), _ptr(v), _ptr(R), _ptr(W_re),
        _ptr(b_re), _ptr(W_v), _ptr(b_v), _ptr(W_role), _ptr(W_l), _ptr(b_l), _ptr(u), float(alpha_role),
        float(alpha_lang), _ptr(packed_v), _ptr(idx), _ptr(k_tok), _ptr(workspace), int(ws_bytes),
        _stream(stream)))


def rolesub_attend_budget(shape, plan: Plan, plan_dev, q, q_strides, K, k_strides, packed_v, idx, k_tok, R,
                          softmax_scale, o, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_attend_budget", lib().rolesub_attend_budget(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(q), *[int(s) for s in q_strides],
        _ptr(K), *[int(s) for s in k_strides], _ptr(packed_v), _ptr(idx), _ptr(k_tok), _ptr(R),
        float(softmax_scale), _ptr(o), _ptr(workspace), int(ws_bytes), _stream(stream)))


def rolesub_attend(shape, plan: Plan, plan_dev, q, q_strides, K, k_strides, packed_v, idx, R,
                   softmax_scale, o, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_attend", lib().rolesub_attend(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(q), *[int(s) for s in q_strides],
        _ptr(K), *[int(s) for s in k_strides], _ptr(packed_v), _ptr(idx), _ptr(R),
        float(softmax_scale), _ptr(o), _ptr(workspace), int(ws_bytes), _stream(stream)))


def rolesub_compress_static(shape, plan: Plan, plan_dev, h, v, R, W_re, b_re, W1, b1, W2, b2,
                            alpha_role, alpha_lang, packed_v, idx, stream=None):
    """rolesub_compress for callers that cannot allocate: the scratch is the
    library's fixed per-GPU array (rolesub_static_scratch_bytes()); no workspace."""
    _check("rolesub_compress_static", lib().rolesub_compress_static(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(h), _ptr(v), _ptr(R), _ptr(W_re),
        _ptr(b_re), _ptr(W1), _ptr(b1), _ptr(W2), _ptr(b2), float(alpha_role), float(alpha_lang),
        _ptr(packed_v), _ptr(idx), _stream(stream)))


def rolesub_static_device_status(stream=None):
    """(code, detail) of the status word the latest rolesub_compress_static
    call left in the fixed array (waits for the stream)."""
    code = ctypes.c_int32(0)
    detail = ctypes.c_int32(0)
    _check("rolesub_static_device_status", lib().rolesub_static_device_status(
        _stream(stream), ctypes.byref(code), ctypes.byref(detail)))
    return code.value, detail.value


def rolesub_static_scratch_bytes():
    """Size of the fixed scratch array compiled into the loaded library."""
    return int(lib().rolesub_static_scratch_bytes())


def rolesub_select_count(n_view, ratio):
    return int(lib().rolesub_select_count(int(n_view), float(ratio)))


def rolesub_select_tokens(scores, x, ratio, keep_idx=None, x_keep=None, stream=None):
    """Token-level reduction: scores [E][V][n] float32, x [E][V][n][hidden]
    (bf16 or float32) on the device; returns keep_idx [E][V][k] int32 and
    x_keep [E][V][k][hidden]."""
    import torch
    E, V, n = scores.shape
    hidden = x.shape[-1]
    k = rolesub_select_count(n, ratio)
    if k < 0:
        raise RoleSubError("rolesub_select_count", 1)
    if keep_idx is None:
        keep_idx = torch.empty((E, V, max(k, 1)), dtype=torch.int32, device=x.device)
    if x_keep is None:
        x_keep = torch.empty((E, V, max(k, 1), hidden), dtype=x.dtype, device=x.device)
    dt = BF16 if x.dtype == torch.bfloat16 else F32
    _check("rolesub_select_tokens", lib().rolesub_select_tokens(
        E, V, n, float(ratio), _ptr(scores), _ptr(x), hidden, dt, _ptr(keep_idx), _ptr(x_keep), _stream(stream)))
    return keep_idx[:, :, :k], x_keep[:, :, :k]


def rolesub_compress_dense(shape, plan: Plan, plan_dev, h, v, R_dense, W_re, b_re, W1, b1, W2, b2, alpha_role,
                           alpha_lang, packed_v, idx, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_compress_dense", lib().rolesub_compress_dense(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(h), _ptr(v), _ptr(R_dense), _ptr(W_re),
        _ptr(b_re), _ptr(W1), _ptr(b1), _ptr(W2), _ptr(b2), float(alpha_role), float(alpha_lang),
        _ptr(packed_v), _ptr(idx), _ptr(workspace), int(ws_bytes), _stream(stream)))


def rolesub_attend_dense(shape, plan: Plan, plan_dev, q, q_strides, K, k_strides, packed_v, idx, R_dense,
                         softmax_scale, o, workspace, ws_bytes=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size() if ws_bytes is None else ws_bytes
    _check("rolesub_attend_dense", lib().rolesub_attend_dense(
        ctypes.byref(shape), plan.host_ptr, _ptr(plan_dev), _ptr(q), *[int(s) for s in q_strides],
        _ptr(K), *[int(s) for s in k_strides], _ptr(packed_v), _ptr(idx), _ptr(R_dense),
        float(softmax_scale), _ptr(o), _ptr(workspace), int(ws_bytes), _stream(stream)))


def rolesub_get_device_status(workspace, stream=None):
    code = ctypes.c_int32(0)
    detail = ctypes.c_int32(0)
    _check("rolesub_get_device_status", lib().rolesub_get_device_status(
        _ptr(workspace), _stream(stream), ctypes.byref(code), ctypes.byref(detail)))
    return code.value, detail.value


def rolesub_reset_device_status(workspace, stream=None):
    _check("rolesub_reset_device_status", lib().rolesub_reset_device_status(_ptr(workspace), _stream(stream)))


def rolesub_wait_selftest(limit_ns, workspace, out, stream=None):
    """Launches the bounded-wait self-test (see the header); out is a device
    int64 tensor of 4 elements."""
    _check("rolesub_wait_selftest", lib().rolesub_wait_selftest(
        int(limit_ns), _ptr(workspace), _ptr(out), _stream(stream)))


def rolesub_status_string(code):
    return lib().rolesub_status_string(int(code)).decode()


def rolesub_version():
    return int(lib().rolesub_version())


def rolesub_launch_count():
    return int(lib().rolesub_launch_count())


# ---------------------------------------------------------------------------
# Convenience wrapper: one cache geometry, resident plan and workspace
# ---------------------------------------------------------------------------

class RoleSub:
    """Holds a shape, its plan (host + device copy) and a workspace.

    compress()/attend() allocate their outputs with torch and call the C
    entry points on the current (or given) stream.
    """

    def __init__(self, L, H, dh, G, C, F, dtype, n_tok, k, n_query, device="cuda"):
        import torch
        self.torch = torch
        self.dtype = dtype
        self.shape = make_shape(L, H, dh, G, C, F, dtype)
        self.plan = Plan(self.shape, n_tok, k, n_query)
        self.plan_dev = self.plan.to_device(device)
        self.ws_bytes = self.plan.workspace_size()
        if dtype in ("bf16", BF16) and dh == 128 and G == 16:
            # room for the per-token budget path's router scores as well
            self.ws_bytes = max(self.ws_bytes, self.plan.budget_workspace_size())
        self.workspace = torch.zeros(self.ws_bytes, dtype=torch.uint8, device=device)
        self.device = device
        self.tdtype = torch.bfloat16 if dtype in ("bf16", BF16) else torch.float32

    def new_outputs(self):
        t = self.torch
        h = self.plan.hdr
        L = self.shape.num_layers
        packed = t.empty((L, max(h.packed_elems_per_layer, 1)), dtype=self.tdtype, device=self.device)
        idx = t.empty((L, max(h.idx_bytes_per_layer, 16)), dtype=t.uint8, device=self.device)
        return packed, idx

    def compress(self, h, v, R, W_re, b_re, W1, b1, W2, b2, alpha_role=0.1, alpha_lang=0.1,
                 packed=None, idx=None, stream=None):
        if packed is None or idx is None:
            packed, idx = self.new_outputs()
        rolesub_compress(self.shape, self.plan, self.plan_dev, h, v, R, W_re, b_re, W1, b1, W2, b2,
                         alpha_role, alpha_lang, packed, idx, self.workspace, self.ws_bytes, stream)
        return packed, idx

    def compress_additive(self, h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l, alpha_role=0.1,
                          alpha_lang=0.1, packed=None, idx=None, stream=None):
        if packed is None or idx is None:
            packed, idx = self.new_outputs()
        rolesub_compress_additive(self.shape, self.plan, self.plan_dev, h, v, R, W_re, b_re, W_v, b_v, W_role,
                                  W_l, b_l, alpha_role, alpha_lang, packed, idx, self.workspace, self.ws_bytes,
                                  stream)
        return packed, idx

    def compress_budget(self, h, v, R, W_re, b_re, W_v, b_v, W_role, W_l, b_l, u, alpha_role=0.1,
                        alpha_lang=0.1, packed=None, idx=None, k_tok=None, stream=None):
        if packed is None or idx is None:
            packed, idx = self.new_outputs()
        if k_tok is None:
            k_tok = self.torch.empty((self.shape.num_layers, max(self.plan.hdr.rows_per_layer, 1)),
                                     dtype=self.torch.uint8, device=self.device)
        rolesub_compress_budget(self.shape, self.plan, self.plan_dev, h, v, R, W_re, b_re, W_v, b_v, W_role, W_l,
                                b_l, u, alpha_role, alpha_lang, packed, idx, k_tok, self.workspace, self.ws_bytes,
                                stream)
        return packed, idx, k_tok

    def attend_budget(self, q, K, packed, idx, k_tok, R, softmax_scale=0.0, o=None, stream=None):
        t = self.torch
        s = self.shape
        d = s.num_heads * s.head_dim
        hdr = self.plan.hdr
        q_strides = (hdr.q_rows_per_layer * d, d, s.head_dim)
        k_strides = (hdr.rows_per_layer * d, d, s.head_dim)
        if o is None:
            o = t.empty((s.num_layers, max(hdr.q_rows_per_layer, 1), d), dtype=self.tdtype, device=self.device)
        rolesub_attend_budget(s, self.plan, self.plan_dev, q, q_strides, K, k_strides, packed, idx, k_tok, R,
                              softmax_scale, o, self.workspace, self.ws_bytes, stream)
        return o

    def _dense_workspace(self):
        if getattr(self, "_dws", None) is None:
            n = self.plan.dense_workspace_size()
            self._dws = self.torch.zeros(n, dtype=self.torch.uint8, device=self.device)
        return self._dws

    def compress_dense(self, h, v, R_dense, W_re, b_re, W1, b1, W2, b2, alpha_role=0.1, alpha_lang=0.1,
                       packed=None, idx=None, stream=None):
        """Dense-rotation compress; the first call allocates its larger
        workspace (one [L][rows][d] bf16 buffer and the pair lists)."""
        if packed is None or idx is None:
            packed, idx = self.new_outputs()
        ws = self._dense_workspace()
        rolesub_compress_dense(self.shape, self.plan, self.plan_dev, h, v, R_dense, W_re, b_re, W1, b1, W2, b2,
                               alpha_role, alpha_lang, packed, idx, ws, ws.numel(), stream)
        return packed, idx

    def attend_dense(self, q, K, packed, idx, R_dense, softmax_scale=0.0, o=None, stream=None):
        t = self.torch
        s = self.shape
        d = s.num_heads * s.head_dim
        hdr = self.plan.hdr
        if o is None:
            o = t.empty((s.num_layers, max(hdr.q_rows_per_layer, 1), d), dtype=self.tdtype, device=self.device)
        ws = self._dense_workspace()
        rolesub_attend_dense(s, self.plan, self.plan_dev, q, (hdr.q_rows_per_layer * d, d, s.head_dim), K,
                             (hdr.rows_per_layer * d, d, s.head_dim), packed, idx, R_dense, softmax_scale, o, ws,
                             ws.numel(), stream)
        return o

    def dense_device_status(self, stream=None):
        return rolesub_get_device_status(self._dense_workspace(), stream)

    def attend(self, q, K, packed, idx, R, softmax_scale=0.0, o=None, q_strides=None, k_strides=None,
               stream=None):
        t = self.torch
        s = self.shape
        d = s.num_heads * s.head_dim
        hdr = self.plan.hdr
        if q_strides is None:
            q_strides = (hdr.q_rows_per_layer * d, d, s.head_dim)
        if k_strides is None:
            k_strides = (hdr.rows_per_layer * d, d, s.head_dim)
        if o is None:
            o = t.empty((s.num_layers, max(hdr.q_rows_per_layer, 1), d), dtype=self.tdtype, device=self.device)
        rolesub_attend(s, self.plan, self.plan_dev, q, q_strides, K, k_strides, packed, idx, R,
                       softmax_scale, o, self.workspace, self.ws_bytes, stream)
        return o

    def device_status(self, stream=None):
        return rolesub_get_device_status(self.workspace, stream)
