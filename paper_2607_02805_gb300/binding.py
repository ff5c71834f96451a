"""ctypes binding of libbdscan (include/bdscan.h): argument marshalling only.

Every function of the C ABI appears here under the same name and takes the
same arguments; the ctypes structures mirror the C structs field by field.
The tensor helpers at the bottom turn torch tensors into those structs (data
pointers, the current CUDA stream) and raise on a non-zero return code. All
computation happens in the CUDA library; if it cannot be loaded, every call
raises. use_debug_build() routes every later call to the debug build of the
same library (device status words, BDSCAN_ERR_DEVICE).
"""

from __future__ import annotations

import ctypes
import os
import threading

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "lib", "libbdscan.so")
LIB_DEBUG_PATH = os.path.join(_HERE, "lib", "libbdscan_debug.so")

BDSCAN_OK = 0
BDSCAN_ERR_ARG = -1
BDSCAN_ERR_UNSUPPORTED = -2
BDSCAN_ERR_CUDA = -3
BDSCAN_ERR_DEVICE = -4
BDSCAN_F32 = 0
BDSCAN_BF16 = 1

c_void_p = ctypes.c_void_p


class bdscan_dims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int64), ("len", ctypes.c_int64), ("block", ctypes.c_int64),
                ("d_inner", ctypes.c_int64), ("d_state", ctypes.c_int64), ("dtype", ctypes.c_int32),
                ("out_dtype", ctypes.c_int32)]


class bdscan_ssd_dims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int64), ("len", ctypes.c_int64), ("block", ctypes.c_int64),
                ("heads", ctypes.c_int64), ("head_dim", ctypes.c_int64), ("d_state", ctypes.c_int64),
                ("dtype", ctypes.c_int32)]


class bdscan_clean(ctypes.Structure):
    _fields_ = [("x", c_void_p), ("dt", c_void_p), ("B", c_void_p), ("C", c_void_p)]


class bdscan_noisy(ctypes.Structure):
    _fields_ = [("x", c_void_p), ("dt_f", c_void_p), ("B_f", c_void_p), ("C_f", c_void_p),
                ("dt_r", c_void_p), ("B_r", c_void_p), ("C_r", c_void_p)]


class bdscan_params(ctypes.Structure):
    _fields_ = [("A_f", c_void_p), ("D_f", c_void_p), ("A_r", c_void_p), ("D_r", c_void_p)]


class bdscan_clean_grads(ctypes.Structure):
    _fields_ = [("dx", c_void_p), ("ddt", c_void_p), ("dB", c_void_p), ("dC", c_void_p)]


class bdscan_noisy_grads(ctypes.Structure):
    _fields_ = [("dx", c_void_p), ("ddt_f", c_void_p), ("dB_f", c_void_p), ("dC_f", c_void_p),
                ("ddt_r", c_void_p), ("dB_r", c_void_p), ("dC_r", c_void_p)]


class bdscan_param_grads(ctypes.Structure):
    _fields_ = [("dA_f", c_void_p), ("dD_f", c_void_p), ("dA_r", c_void_p), ("dD_r", c_void_p)]


class bdscan_mixer_params(ctypes.Structure):
    _fields_ = [("conv_w", c_void_p), ("conv_b", c_void_p), ("dt_bias_f", c_void_p), ("dt_bias_r", c_void_p)]


class bdscan_mixer_grads(ctypes.Structure):
    _fields_ = [("dconv_w", c_void_p), ("dconv_b", c_void_p), ("ddt_bias_f", c_void_p), ("ddt_bias_r", c_void_p)]


class bdscan_adaln(ctypes.Structure):
    _fields_ = [("shift", c_void_p), ("scale", c_void_p), ("gate", c_void_p), ("eps", ctypes.c_float)]


# (name, restype, argtypes) of every exported function, in header order
_P = ctypes.POINTER
SIGNATURES = [
    ("bdscan_last_error", ctypes.c_char_p, []),
    ("bdscan_version", ctypes.c_int, []),
    ("bdscan_chunk_tokens", ctypes.c_int64, [ctypes.c_int64]),
    ("bdscan_profile_events", ctypes.c_int, [ctypes.POINTER(c_void_p), ctypes.c_int]),
    ("bdscan_last_launch_count", ctypes.c_int, []),
    ("bdscan_forward_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_forward", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p, c_void_p,
      c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_backward_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_backward", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p, c_void_p,
      c_void_p, _P(bdscan_clean_grads), _P(bdscan_noisy_grads), _P(bdscan_param_grads), c_void_p,
      ctypes.c_size_t, c_void_p]),
    ("bdscan_boundary_states_workspace_size", ctypes.c_size_t, [_P(bdscan_dims), ctypes.c_int]),
    ("bdscan_boundary_states", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, ctypes.c_int,
      c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_active_block", ctypes.c_int,
     [_P(bdscan_dims), c_void_p, _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p]),
    ("bdscan_active_block_adaln_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_active_block_adaln", ctypes.c_int,
     [_P(bdscan_dims), c_void_p, _P(bdscan_noisy), _P(bdscan_params), _P(bdscan_adaln), c_void_p, c_void_p,
      ctypes.c_size_t, c_void_p]),
    ("bdscan_boundary_states_noalloc", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, ctypes.c_int, c_void_p]),
    ("bdscan_full_bidir_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_full_bidir_forward", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_mixer_forward_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_mixer_forward", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), c_void_p, _P(bdscan_noisy), c_void_p, _P(bdscan_params),
      _P(bdscan_mixer_params), c_void_p, c_void_p, c_void_p, c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_mixer_backward_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_mixer_backward", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), c_void_p, _P(bdscan_noisy), c_void_p, _P(bdscan_params),
      _P(bdscan_mixer_params), c_void_p, c_void_p, c_void_p, _P(bdscan_clean_grads), c_void_p,
      _P(bdscan_noisy_grads), c_void_p, _P(bdscan_param_grads), _P(bdscan_mixer_grads), c_void_p, ctypes.c_size_t,
      c_void_p]),
    ("bdscan_mixer_boundary_states_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_mixer_boundary_states", ctypes.c_int,
     [_P(bdscan_dims), _P(bdscan_clean), c_void_p, c_void_p, c_void_p, _P(bdscan_mixer_params), c_void_p, c_void_p,
      c_void_p, c_void_p, c_void_p, ctypes.c_int, c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_mixer_active_block_workspace_size", ctypes.c_size_t, [_P(bdscan_dims)]),
    ("bdscan_mixer_active_block", ctypes.c_int,
     [_P(bdscan_dims), c_void_p, c_void_p, _P(bdscan_noisy), c_void_p, _P(bdscan_params), _P(bdscan_mixer_params),
      c_void_p, c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_ssd_forward_workspace_size", ctypes.c_size_t, [_P(bdscan_ssd_dims)]),
    ("bdscan_ssd_forward", ctypes.c_int,
     [_P(bdscan_ssd_dims), _P(bdscan_clean), _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p, c_void_p,
      c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_ssd_boundary_states_workspace_size", ctypes.c_size_t, [_P(bdscan_ssd_dims), ctypes.c_int]),
    ("bdscan_ssd_boundary_states", ctypes.c_int,
     [_P(bdscan_ssd_dims), _P(bdscan_clean), c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, ctypes.c_int,
      c_void_p, ctypes.c_size_t, c_void_p]),
    ("bdscan_ssd_active_block", ctypes.c_int,
     [_P(bdscan_ssd_dims), c_void_p, _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p]),
    ("bdscan_ssd_backward_workspace_size", ctypes.c_size_t, [_P(bdscan_ssd_dims)]),
    ("bdscan_ssd_backward", ctypes.c_int,
     [_P(bdscan_ssd_dims), _P(bdscan_clean), _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p, c_void_p,
      c_void_p, _P(bdscan_clean_grads), _P(bdscan_noisy_grads), _P(bdscan_param_grads), c_void_p, ctypes.c_size_t,
      c_void_p]),
    ("bdscan_ssd_wait_flag", ctypes.c_int, [ctypes.c_int]),
    ("bdscan_debug_build", ctypes.c_int, []),
    ("bdscan_debug_set_slack", ctypes.c_int, [ctypes.c_longlong]),
    ("bdscan_ssd_wait_selftest", ctypes.c_int, [ctypes.c_uint32]),
    ("bdscan_ssd_tma_enabled", ctypes.c_int, []),
    ("bdscan_ssd_set_tma", ctypes.c_int, [ctypes.c_int]),
    ("bdscan_ssd_full_bidir_workspace_size", ctypes.c_size_t, [_P(bdscan_ssd_dims)]),
    ("bdscan_ssd_full_bidir_forward", ctypes.c_int,
     [_P(bdscan_ssd_dims), _P(bdscan_noisy), _P(bdscan_params), c_void_p, c_void_p, ctypes.c_size_t, c_void_p]),
]

BDSCAN_NOALLOC_SCRATCH_BYTES = 32 << 20

_lock = threading.Lock()
_libs = {False: None, True: None}
_use_debug = False


def load(build_if_missing: bool = True, debug=None):
    """Load the CUDA library (building it in-tree first if it is missing or
    stale): the release build, or the debug build when `debug` is true (by
    default the one use_debug_build() selected)."""
    dbg = _use_debug if debug is None else bool(debug)
    path = LIB_DEBUG_PATH if dbg else LIB_PATH
    with _lock:
        if _libs[dbg] is None:
            if build_if_missing:
                from . import build as _build
                _build.build(debug=dbg)
            if not os.path.exists(path):
                raise RuntimeError(f"libbdscan is not built ({path} missing); run paper_2607_02805_gb300/build.py")
            lib = ctypes.CDLL(path)
            for name, res, args in SIGNATURES:
                f = getattr(lib, name)
                f.restype = res
                f.argtypes = args
            _libs[dbg] = lib
    return _libs[dbg]


def use_debug_build(on: bool = True) -> None:
    """Route every later call of this module to the debug build (or back)."""
    global _use_debug
    if on:
        load(debug=True)
    _use_debug = bool(on)


class BdscanError(RuntimeError):
    def __init__(self, fn, code, msg):
        super().__init__(f"{fn} failed with code {code}: {msg}")
        self.code = code


def _call(name, *args):
    lib = load()
    rc = getattr(lib, name)(*args)
    if rc != BDSCAN_OK:
        raise BdscanError(name, rc, lib.bdscan_last_error().decode())
    return rc


def _ref(x):
    return None if x is None else ctypes.byref(x)


# raw functions, same names and arguments as the C ABI
def bdscan_last_error() -> str:
    return load().bdscan_last_error().decode()


def bdscan_debug_build() -> int:
    return load().bdscan_debug_build()


def bdscan_debug_set_slack(elements) -> int:
    return load().bdscan_debug_set_slack(elements)


def bdscan_version() -> int:
    return load().bdscan_version()


def bdscan_chunk_tokens(block: int) -> int:
    return load().bdscan_chunk_tokens(block)


def bdscan_profile_events(events, n) -> int:
    """events: a ctypes array of c_void_p (cudaEvent_t handles) or None."""
    return load().bdscan_profile_events(events, int(n))


def bdscan_last_launch_count() -> int:
    return load().bdscan_last_launch_count()


def bdscan_forward_workspace_size(dims) -> int:
    return load().bdscan_forward_workspace_size(_ref(dims))


def bdscan_backward_workspace_size(dims) -> int:
    return load().bdscan_backward_workspace_size(_ref(dims))


def bdscan_boundary_states_workspace_size(dims, emit_all) -> int:
    return load().bdscan_boundary_states_workspace_size(_ref(dims), int(emit_all))


def bdscan_forward(dims, clean, noisy, params, y_c, y_n, states, workspace, workspace_bytes, stream):
    return load().bdscan_forward(_ref(dims), _ref(clean), _ref(noisy),
                                 _ref(params), y_c, y_n, states, workspace, workspace_bytes, stream)


def bdscan_backward(dims, clean, noisy, params, states, dy_c, dy_n, dstates, gclean, gnoisy, gparams,
                    workspace, workspace_bytes, stream):
    return load().bdscan_backward(_ref(dims), _ref(clean), _ref(noisy),
                                  _ref(params), states, dy_c, dy_n, dstates, _ref(gclean),
                                  _ref(gnoisy), _ref(gparams), workspace, workspace_bytes, stream)


def bdscan_boundary_states(dims, clean, A_f, D_f, init_state, y_c, states, emit_all, workspace,
                           workspace_bytes, stream):
    return load().bdscan_boundary_states(_ref(dims), _ref(clean), A_f, D_f, init_state, y_c,
                                         states, int(emit_all), workspace, workspace_bytes, stream)


def bdscan_active_block(dims, seed, noisy, params, y_n, stream):
    return load().bdscan_active_block(_ref(dims), seed, _ref(noisy), _ref(params),
                                      y_n, stream)


def bdscan_active_block_adaln_workspace_size(dims) -> int:
    return load().bdscan_active_block_adaln_workspace_size(_ref(dims))


def bdscan_active_block_adaln(dims, seed, noisy, params, mod, out, workspace, workspace_bytes, stream):
    return load().bdscan_active_block_adaln(_ref(dims), seed, _ref(noisy), _ref(params), _ref(mod), out,
                                            workspace, workspace_bytes, stream)


def bdscan_boundary_states_noalloc(dims, clean, A_f, D_f, init_state, y_c, states, emit_all, stream):
    return load().bdscan_boundary_states_noalloc(_ref(dims), _ref(clean), A_f, D_f, init_state, y_c, states,
                                                 int(emit_all), stream)


def bdscan_full_bidir_workspace_size(dims) -> int:
    return load().bdscan_full_bidir_workspace_size(_ref(dims))


def bdscan_full_bidir_forward(dims, noisy, params, y, workspace, workspace_bytes, stream):
    return load().bdscan_full_bidir_forward(_ref(dims), _ref(noisy), _ref(params), y, workspace,
                                            workspace_bytes, stream)


def bdscan_mixer_forward_workspace_size(dims) -> int:
    return load().bdscan_mixer_forward_workspace_size(_ref(dims))


def bdscan_mixer_forward(dims, clean, z_c, noisy, z_n, params, mparams, out_c, out_n, states, workspace,
                         workspace_bytes, stream):
    return load().bdscan_mixer_forward(_ref(dims), _ref(clean), z_c, _ref(noisy), z_n, _ref(params), _ref(mparams),
                                       out_c, out_n, states, workspace, workspace_bytes, stream)


def bdscan_mixer_backward_workspace_size(dims) -> int:
    return load().bdscan_mixer_backward_workspace_size(_ref(dims))


def bdscan_mixer_backward(dims, clean, z_c, noisy, z_n, params, mparams, dout_c, dout_n, dstates, gclean, dz_c,
                          gnoisy, dz_n, gparams, gmparams, workspace, workspace_bytes, stream):
    return load().bdscan_mixer_backward(_ref(dims), _ref(clean), z_c, _ref(noisy), z_n, _ref(params), _ref(mparams),
                                        dout_c, dout_n, dstates, _ref(gclean), dz_c, _ref(gnoisy), dz_n,
                                        _ref(gparams), _ref(gmparams), workspace, workspace_bytes, stream)


def bdscan_mixer_boundary_states_workspace_size(dims) -> int:
    return load().bdscan_mixer_boundary_states_workspace_size(_ref(dims))


def bdscan_mixer_boundary_states(dims, clean, z_c, A_f, D_f, mparams, init_state, conv_init, out_c, states,
                                 conv_states, emit_all, workspace, workspace_bytes, stream):
    return load().bdscan_mixer_boundary_states(_ref(dims), _ref(clean), z_c, A_f, D_f, _ref(mparams), init_state,
                                               conv_init, out_c, states, conv_states, int(emit_all), workspace,
                                               workspace_bytes, stream)


def bdscan_mixer_active_block_workspace_size(dims) -> int:
    return load().bdscan_mixer_active_block_workspace_size(_ref(dims))


def bdscan_mixer_active_block(dims, seed, conv_seed, noisy, z_n, params, mparams, out_n, workspace, workspace_bytes,
                              stream):
    return load().bdscan_mixer_active_block(_ref(dims), seed, conv_seed, _ref(noisy), z_n, _ref(params),
                                            _ref(mparams), out_n, workspace, workspace_bytes, stream)


def bdscan_ssd_forward_workspace_size(dims) -> int:
    return load().bdscan_ssd_forward_workspace_size(_ref(dims))


def bdscan_ssd_forward(dims, clean, noisy, params, y_c, y_n, states, workspace, workspace_bytes, stream):
    return load().bdscan_ssd_forward(_ref(dims), _ref(clean), _ref(noisy), _ref(params), y_c, y_n, states,
                                     workspace, workspace_bytes, stream)


def bdscan_ssd_boundary_states_workspace_size(dims, emit_all) -> int:
    return load().bdscan_ssd_boundary_states_workspace_size(_ref(dims), int(emit_all))


def bdscan_ssd_boundary_states(dims, clean, A_f, D_f, init_state, y_c, states, emit_all, workspace,
                               workspace_bytes, stream):
    return load().bdscan_ssd_boundary_states(_ref(dims), _ref(clean), A_f, D_f, init_state, y_c, states,
                                             int(emit_all), workspace, workspace_bytes, stream)


def bdscan_ssd_active_block(dims, seed, noisy, params, y_n, stream):
    return load().bdscan_ssd_active_block(_ref(dims), seed, _ref(noisy), _ref(params), y_n, stream)


def bdscan_ssd_backward_workspace_size(dims) -> int:
    return load().bdscan_ssd_backward_workspace_size(_ref(dims))


def bdscan_ssd_backward(dims, clean, noisy, params, states, dy_c, dy_n, dstates, gclean, gnoisy, gparams, workspace,
                        workspace_bytes, stream):
    return load().bdscan_ssd_backward(_ref(dims), _ref(clean), _ref(noisy), _ref(params), states, dy_c, dy_n, dstates,
                                      _ref(gclean), _ref(gnoisy), _ref(gparams), workspace, workspace_bytes, stream)


def bdscan_ssd_wait_flag(reset) -> int:
    return load().bdscan_ssd_wait_flag(int(reset))


def bdscan_ssd_wait_selftest(polls) -> int:
    return load().bdscan_ssd_wait_selftest(int(polls))


def bdscan_ssd_tma_enabled() -> int:
    return load().bdscan_ssd_tma_enabled()


def bdscan_ssd_set_tma(enable) -> int:
    return load().bdscan_ssd_set_tma(int(enable))


def bdscan_ssd_full_bidir_workspace_size(dims) -> int:
    return load().bdscan_ssd_full_bidir_workspace_size(_ref(dims))


def bdscan_ssd_full_bidir_forward(dims, noisy, params, y, workspace, workspace_bytes, stream):
    return load().bdscan_ssd_full_bidir_forward(_ref(dims), _ref(noisy), _ref(params), y, workspace,
                                                workspace_bytes, stream)

# ---------------------------------------------------------------------------
# torch-tensor helpers (marshalling only)
# ---------------------------------------------------------------------------
def _ptr(t):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("bdscan tensors must be contiguous")
    return t.data_ptr()


def _stream(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def _dtype_code(t):
    import torch
    if t.dtype == torch.float32:
        return BDSCAN_F32
    if t.dtype == torch.bfloat16:
        return BDSCAN_BF16
    raise ValueError(f"unsupported dtype {t.dtype}")


def make_dims(batch, length, block, d_inner, d_state, dtype, out_dtype=None):
    return bdscan_dims(int(batch), int(length), int(block), int(d_inner), int(d_state), int(dtype),
                       int(dtype if out_dtype is None else out_dtype))


def make_clean(t):
    return bdscan_clean(_ptr(t["x_c"]), _ptr(t["dt_c"]), _ptr(t["B_c"]), _ptr(t["C_c"]))


def make_noisy(t):
    return bdscan_noisy(_ptr(t["x_n"]), _ptr(t["dt_f"]), _ptr(t["B_f"]), _ptr(t["C_f"]), _ptr(t["dt_r"]),
                        _ptr(t["B_r"]), _ptr(t["C_r"]))


def make_params(t):
    return bdscan_params(_ptr(t["A_f"]), _ptr(t["D_f"]), _ptr(t["A_r"]), _ptr(t["D_r"]))


def forward(dims, t, y_c, y_n, states, workspace, stream=None):
    """t: dict of device tensors keyed like paper_2607_02805_gb300.inputs."""
    _call("bdscan_forward", ctypes.byref(dims), ctypes.byref(make_clean(t)), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(y_c), _ptr(y_n), _ptr(states), _ptr(workspace),
          workspace.numel() * workspace.element_size(), _stream(stream))


def backward(dims, t, states, dy_c, dy_n, dstates, g, workspace, stream=None):
    """g: dict of gradient tensors keyed by input name (x_c, ..., D_r)."""
    gc = bdscan_clean_grads(_ptr(g["x_c"]), _ptr(g["dt_c"]), _ptr(g["B_c"]), _ptr(g["C_c"]))
    gn = bdscan_noisy_grads(_ptr(g["x_n"]), _ptr(g["dt_f"]), _ptr(g["B_f"]), _ptr(g["C_f"]), _ptr(g["dt_r"]),
                            _ptr(g["B_r"]), _ptr(g["C_r"]))
    gp = bdscan_param_grads(_ptr(g["A_f"]), _ptr(g["D_f"]), _ptr(g["A_r"]), _ptr(g["D_r"]))
    _call("bdscan_backward", ctypes.byref(dims), ctypes.byref(make_clean(t)), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(states), _ptr(dy_c), _ptr(dy_n), _ptr(dstates), ctypes.byref(gc),
          ctypes.byref(gn), ctypes.byref(gp), _ptr(workspace), workspace.numel() * workspace.element_size(),
          _stream(stream))


def boundary_states(dims, t, init_state, y_c, states, emit_all, workspace, stream=None):
    _call("bdscan_boundary_states", ctypes.byref(dims), ctypes.byref(make_clean(t)), _ptr(t["A_f"]),
          _ptr(t["D_f"]), _ptr(init_state), _ptr(y_c), _ptr(states), int(emit_all), _ptr(workspace),
          0 if workspace is None else workspace.numel() * workspace.element_size(), _stream(stream))


def active_block(dims, seed, t, y_n, stream=None):
    _call("bdscan_active_block", ctypes.byref(dims), _ptr(seed), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(y_n), _stream(stream))


def active_block_adaln(dims, seed, t, shift, scale, gate, eps, out, workspace, stream=None):
    """One timestep-modulated active block: t["x_n"] is the block's hidden input
    h; out = h + gate * y_n of the modulated input."""
    mod = bdscan_adaln(_ptr(shift), _ptr(scale), _ptr(gate), float(eps))
    _call("bdscan_active_block_adaln", ctypes.byref(dims), _ptr(seed), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), ctypes.byref(mod), _ptr(out), _ptr(workspace),
          0 if workspace is None else workspace.numel() * workspace.element_size(), _stream(stream))


def full_bidir_forward(dims, t, y, workspace, stream=None):
    """Full-sequence bidirectional layer (no block restriction) of the noisy
    tensors in t; y [Bt][L][D]."""
    _call("bdscan_full_bidir_forward", ctypes.byref(dims), ctypes.byref(make_noisy(t)), ctypes.byref(make_params(t)),
          _ptr(y), _ptr(workspace), 0 if workspace is None else workspace.numel() * workspace.element_size(),
          _stream(stream))


def make_ssd_dims(batch, length, block, heads, d_state, head_dim=64):
    return bdscan_ssd_dims(int(batch), int(length), int(block), int(heads), int(head_dim), int(d_state),
                           BDSCAN_BF16)


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def ssd_forward(dims, t, y_c, y_n, states, workspace, stream=None):
    """SSD-form all-block forward; t holds the tensors in the layouts of
    include/bdscan_ssd.h, keyed like the diagonal layer's (x_c, ..., D_r)."""
    _call("bdscan_ssd_forward", ctypes.byref(dims), ctypes.byref(make_clean(t)), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(y_c), _ptr(y_n), _ptr(states), _ptr(workspace), _nbytes(workspace),
          _stream(stream))


def ssd_boundary_states(dims, t, init_state, y_c, states, emit_all, workspace, stream=None):
    _call("bdscan_ssd_boundary_states", ctypes.byref(dims), ctypes.byref(make_clean(t)), _ptr(t["A_f"]),
          _ptr(t["D_f"]), _ptr(init_state), _ptr(y_c), _ptr(states), int(emit_all), _ptr(workspace),
          _nbytes(workspace), _stream(stream))


def ssd_active_block(dims, seed, t, y_n, stream=None):
    _call("bdscan_ssd_active_block", ctypes.byref(dims), _ptr(seed), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(y_n), _stream(stream))


def ssd_full_bidir_forward(dims, t, y, workspace, stream=None):
    """Full-sequence bidirectional SSD layer (no block restriction) of the noisy
    tensors in t; y [Bt][L][H][64]."""
    _call("bdscan_ssd_full_bidir_forward", ctypes.byref(dims), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(y), _ptr(workspace), _nbytes(workspace), _stream(stream))


# ---------------------------------------------------------------------------
# mixer (include/bdscan_mixer.h): tensors keyed xr_c, dtr_c, B_c, C_c, z_c,
# xr_n, dtr_f, B_f, C_f, dtr_r, B_r, C_r, z_n, A_f, D_f, A_r, D_r, conv_w,
# conv_b, dt_bias_f, dt_bias_r
# ---------------------------------------------------------------------------
def make_mixer_params(t):
    return bdscan_mixer_params(_ptr(t["conv_w"]), _ptr(t["conv_b"]), _ptr(t["dt_bias_f"]), _ptr(t["dt_bias_r"]))


def _mix_clean(t):
    return bdscan_clean(_ptr(t["xr_c"]), _ptr(t["dtr_c"]), _ptr(t["B_c"]), _ptr(t["C_c"]))


def _mix_noisy(t):
    return bdscan_noisy(_ptr(t["xr_n"]), _ptr(t["dtr_f"]), _ptr(t["B_f"]), _ptr(t["C_f"]), _ptr(t["dtr_r"]),
                        _ptr(t["B_r"]), _ptr(t["C_r"]))


def mixer_forward(dims, t, out_c, out_n, states, workspace, stream=None):
    _call("bdscan_mixer_forward", ctypes.byref(dims), ctypes.byref(_mix_clean(t)), _ptr(t["z_c"]),
          ctypes.byref(_mix_noisy(t)), _ptr(t["z_n"]), ctypes.byref(make_params(t)),
          ctypes.byref(make_mixer_params(t)), _ptr(out_c), _ptr(out_n), _ptr(states), _ptr(workspace),
          _nbytes(workspace), _stream(stream))


def mixer_backward(dims, t, dout_c, dout_n, dstates, g, workspace, stream=None):
    """g: gradient tensors keyed like t (xr_c ... z_n, A_f ... dt_bias_r)."""
    gc = bdscan_clean_grads(_ptr(g["xr_c"]), _ptr(g["dtr_c"]), _ptr(g["B_c"]), _ptr(g["C_c"]))
    gn = bdscan_noisy_grads(_ptr(g["xr_n"]), _ptr(g["dtr_f"]), _ptr(g["B_f"]), _ptr(g["C_f"]), _ptr(g["dtr_r"]),
                            _ptr(g["B_r"]), _ptr(g["C_r"]))
    gp = bdscan_param_grads(_ptr(g["A_f"]), _ptr(g["D_f"]), _ptr(g["A_r"]), _ptr(g["D_r"]))
    gm = bdscan_mixer_grads(_ptr(g["conv_w"]), _ptr(g["conv_b"]), _ptr(g["dt_bias_f"]), _ptr(g["dt_bias_r"]))
    _call("bdscan_mixer_backward", ctypes.byref(dims), ctypes.byref(_mix_clean(t)), _ptr(t["z_c"]),
          ctypes.byref(_mix_noisy(t)), _ptr(t["z_n"]), ctypes.byref(make_params(t)),
          ctypes.byref(make_mixer_params(t)), _ptr(dout_c), _ptr(dout_n), _ptr(dstates), ctypes.byref(gc),
          _ptr(g["z_c"]), ctypes.byref(gn), _ptr(g["z_n"]), ctypes.byref(gp), ctypes.byref(gm), _ptr(workspace),
          _nbytes(workspace), _stream(stream))


def mixer_boundary_states(dims, t, init_state, conv_init, out_c, states, conv_states, emit_all, workspace,
                          stream=None):
    _call("bdscan_mixer_boundary_states", ctypes.byref(dims), ctypes.byref(_mix_clean(t)),
          _ptr(t["z_c"]) if out_c is not None else None, _ptr(t["A_f"]), _ptr(t["D_f"]),
          ctypes.byref(make_mixer_params(t)), _ptr(init_state), _ptr(conv_init), _ptr(out_c), _ptr(states),
          _ptr(conv_states), int(emit_all), _ptr(workspace), _nbytes(workspace), _stream(stream))


def mixer_active_block(dims, seed, conv_seed, t, out_n, workspace, stream=None):
    _call("bdscan_mixer_active_block", ctypes.byref(dims), _ptr(seed), _ptr(conv_seed), ctypes.byref(_mix_noisy(t)),
          _ptr(t["z_n"]), ctypes.byref(make_params(t)), ctypes.byref(make_mixer_params(t)), _ptr(out_n),
          _ptr(workspace), _nbytes(workspace), _stream(stream))


def ssd_backward(dims, t, states, dy_c, dy_n, dstates, g, workspace, stream=None):
    """SSD-form backward; g holds the gradient tensors keyed like t."""
    gc = bdscan_clean_grads(_ptr(g["x_c"]), _ptr(g["dt_c"]), _ptr(g["B_c"]), _ptr(g["C_c"]))
    gn = bdscan_noisy_grads(_ptr(g["x_n"]), _ptr(g["dt_f"]), _ptr(g["B_f"]), _ptr(g["C_f"]), _ptr(g["dt_r"]),
                            _ptr(g["B_r"]), _ptr(g["C_r"]))
    gp = bdscan_param_grads(_ptr(g["A_f"]), _ptr(g["D_f"]), _ptr(g["A_r"]), _ptr(g["D_r"]))
    _call("bdscan_ssd_backward", ctypes.byref(dims), ctypes.byref(make_clean(t)), ctypes.byref(make_noisy(t)),
          ctypes.byref(make_params(t)), _ptr(states), _ptr(dy_c), _ptr(dy_n), _ptr(dstates), ctypes.byref(gc),
          ctypes.byref(gn), ctypes.byref(gp), _ptr(workspace), _nbytes(workspace), _stream(stream))
