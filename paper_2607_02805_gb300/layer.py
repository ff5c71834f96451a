"""Device-resident state for repeated calls of the C ABI from PyTorch.

PyTorch provides the device memory and the stream; every step of the scan
runs in libbdscan through ``binding``. A ``Layer`` holds one problem's
inputs, outputs, saved boundary states, gradients and workspaces.
"""

from __future__ import annotations

import numpy as np
import torch

from . import binding
from .inputs import PARAMS, TOKEN_D, TOKEN_N

GRAD_KEYS = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r",
             "A_f", "D_f", "A_r", "D_r")


def to_device(a: np.ndarray, dtype_code: int, device) -> torch.Tensor:
    """uint16 bf16 bits -> torch.bfloat16; float32 stays float32."""
    if a.dtype == np.uint16:
        t = torch.from_numpy(a.view(np.int16).copy()).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(device).contiguous()


def to_numpy(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


class Layer:
    def __init__(self, wl, out_dtype=None, device="cuda", with_dstates=False):
        self.wl = wl
        self.device = torch.device(device)
        dt = binding.BDSCAN_BF16 if wl.dtype == "bf16" else binding.BDSCAN_F32
        od = dt if out_dtype is None else out_dtype
        self.dims = binding.make_dims(wl.batch, wl.len, wl.block, wl.d_inner, wl.d_state, dt, od)
        self.in_torch = torch.bfloat16 if dt == binding.BDSCAN_BF16 else torch.float32
        self.out_torch = torch.bfloat16 if od == binding.BDSCAN_BF16 else torch.float32
        self.t = {k: to_device(wl.dev_bits(k), dt, self.device) for k in wl.t32}
        Bt, L, D, N = wl.batch, wl.len, wl.d_inner, wl.d_state
        nb = L // wl.block
        z = lambda shape, dtyp: torch.zeros(shape, dtype=dtyp, device=self.device)
        self.y_c = z((Bt, L, D), self.out_torch)
        self.y_n = z((Bt, L, D), self.out_torch)
        self.states = z((Bt, nb, D, N), torch.float32)
        self.ws_f = z((max(1, binding.bdscan_forward_workspace_size(self.dims)) + 3) // 4, torch.float32)
        self.ws_b = None
        self.g = None

    def forward(self, stream=None):
        binding.forward(self.dims, self.t, self.y_c, self.y_n, self.states, self.ws_f, stream)

    def alloc_backward(self):
        wl = self.wl
        Bt, L, D, N = wl.batch, wl.len, wl.d_inner, wl.d_state
        self.ws_b = torch.zeros((max(1, binding.bdscan_backward_workspace_size(self.dims)) + 3) // 4,
                                dtype=torch.float32, device=self.device)
        g = {}
        for k in GRAD_KEYS:
            if k in PARAMS:
                g[k] = torch.zeros(self.t[k].shape, dtype=torch.float32, device=self.device)
            else:
                g[k] = torch.zeros(self.t[k].shape, dtype=self.out_torch, device=self.device)
        self.g = g

    def backward(self, stream=None, use_dy_c=True, use_dstates=None):
        if self.g is None:
            self.alloc_backward()
        dstates = self.t.get("dstates") if use_dstates is None or use_dstates else None
        if use_dstates is None:
            dstates = self.t.get("dstates")
        binding.backward(self.dims, self.t, self.states, self.t["dy_c"] if use_dy_c else None, self.t["dy_n"],
                         dstates, self.g, self.ws_b, stream)
