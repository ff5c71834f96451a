"""fp64 CPU oracle for the block-restricted bidirectional selective scan.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline of ``bench.py`` may import this package. It is independent of the
CUDA library: it neither imports ``paper_2607_02805_gb300`` nor shares any of
its code, and the CUDA path never calls it.

The arithmetic lives in ``bdscan_oracle.c`` (plain C, fp64, one loop per
recurrence of the paper); this module builds it with gcc and wraps it with
ctypes. Every function takes numpy arrays (any float dtype, converted to
fp64) in the layouts documented in the C file and returns fp64 arrays.

Parity status of each function (pins live in ``tests/test_oracle_pins.py``):
  forward, boundary_states, active_block -- pinned by the explicit
      semiseparable-matrix brute force, closed forms (block size 1, dt = 0,
      x = 0), the seed-indexing and single-block invariants and bit-exact
      caching;
  backward -- pinned by central finite differences of the pinned forward and
      by the exact transpose of the matrix form for dx.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bdscan_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


class _Dims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_long), ("len", ctypes.c_long), ("block", ctypes.c_long),
                ("d", ctypes.c_long), ("n", ctypes.c_long)]


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/liboracle.so`` (gcc, OpenMP)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
           "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            P = ctypes.c_void_p
            lib.bdo_forward.argtypes = [ctypes.POINTER(_Dims)] + [P] * 18
            lib.bdo_boundary_states.argtypes = [ctypes.POINTER(_Dims)] + [P] * 9 + [ctypes.c_int]
            lib.bdo_active_block.argtypes = [ctypes.POINTER(_Dims)] + [P] * 13
            lib.bdo_backward.argtypes = [ctypes.POINTER(_Dims)] + [P] * 34
            for f in (lib.bdo_forward, lib.bdo_boundary_states, lib.bdo_active_block, lib.bdo_backward):
                f.restype = ctypes.c_int
            lib.bdo_set_threads.argtypes = [ctypes.c_int]
            lib.bdo_get_threads.restype = ctypes.c_int
            lib.bdo_has_openmp.restype = ctypes.c_int
            _lib = lib
    return _lib


def set_threads(n: int) -> None:
    _load().bdo_set_threads(int(n))


def get_threads() -> int:
    return int(_load().bdo_get_threads())


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dims(batch, length, block, d, n):
    return _Dims(int(batch), int(length), int(block), int(d), int(n))


def _check(rc, name):
    if rc != 0:
        raise ValueError(f"oracle {name}: bad arguments (rc={rc})")


def forward(block, x_c, dt_c, B_c, C_c, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r):
    """All-block forward. Returns (y_c, y_n, states[Bt, L/Bs, D, N])."""
    lib = _load()
    ins = [_f64(a) for a in (x_c, dt_c, B_c, C_c, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r)]
    Bt, L, D = ins[0].shape
    N = ins[2].shape[2]
    nb = L // block if block > 0 else 0
    y_c = np.zeros((Bt, L, D))
    y_n = np.zeros((Bt, L, D))
    st = np.zeros((Bt, nb, D, N))
    m = _dims(Bt, L, block, D, N)
    _check(lib.bdo_forward(ctypes.byref(m), *[_p(a) for a in ins], _p(y_c), _p(y_n), _p(st)), "forward")
    return y_c, y_n, st


def boundary_states(block, x_c, dt_c, B_c, C_c, A_f, D_f, init_state=None, emit_all=True, want_y=False):
    """Cache build. Returns (states, y_c or None); states is [Bt, L/Bs or 1, D, N]."""
    lib = _load()
    ins = [_f64(a) for a in (x_c, dt_c, B_c, C_c, A_f, D_f)]
    Bt, L, D = ins[0].shape
    N = ins[2].shape[2]
    nS = (L // block) if emit_all else 1
    st = np.zeros((Bt, nS, D, N))
    y = np.zeros((Bt, L, D)) if want_y else None
    init = None if init_state is None else _f64(init_state)
    m = _dims(Bt, L, block, D, N)
    _check(lib.bdo_boundary_states(ctypes.byref(m), *[_p(a) for a in ins], _p(init), _p(y), _p(st),
                                   1 if emit_all else 0), "boundary_states")
    return st, y


def active_block(seed, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r):
    """One cached noisy block (its length is the block size). Returns y_n."""
    lib = _load()
    ins = [_f64(a) for a in (seed, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r)]
    Bt, Bs, D = ins[1].shape
    N = ins[3].shape[2]
    y_n = np.zeros((Bt, Bs, D))
    m = _dims(Bt, Bs, Bs, D, N)
    _check(lib.bdo_active_block(ctypes.byref(m), *[_p(a) for a in ins], _p(y_n)), "active_block")
    return y_n


GRAD_NAMES = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r",
              "A_f", "D_f", "A_r", "D_r")


def backward(block, x_c, dt_c, B_c, C_c, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r,
             states, dy_c, dy_n, dstates=None):
    """Gradients of <dy_c,y_c> + <dy_n,y_n> + <dstates,states>. Returns a dict
    keyed by input name ("x_c", ..., "D_r"); dy_c and dstates may be None."""
    lib = _load()
    ins = [_f64(a) for a in (x_c, dt_c, B_c, C_c, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r)]
    Bt, L, D = ins[0].shape
    N = ins[2].shape[2]
    st = _f64(states)
    dyc = None if dy_c is None else _f64(dy_c)
    dyn = _f64(dy_n)
    dst = None if dstates is None else _f64(dstates)
    out = {k: np.zeros_like(v) for k, v in zip(GRAD_NAMES, ins)}
    m = _dims(Bt, L, block, D, N)
    _check(lib.bdo_backward(ctypes.byref(m), *[_p(a) for a in ins], _p(st), _p(dyc), _p(dyn), _p(dst),
                            *[_p(out[k]) for k in GRAD_NAMES]), "backward")
    return out
