"""Seeded synthetic inputs for the block-restricted bidirectional selective scan.

This module is shared by the tests, the benchmark and the oracle checks. It
holds random-number generation and number-format conversion only: none of the
scan's arithmetic lives here.

Workload recipe (the paper trains on DCLM text through trained models; these
synthetic draws stand in for the activations such a model feeds one Mamba
layer, with the value ranges of a Mamba-1 style parameterisation):

* x ~ N(0, 1)                       per token and channel, [Bt, L, D]
* dt = softplus(N(-2, 0.5))         per token and channel, [Bt, L, D]
  (the step size is given after its softplus, median about 0.13)
* B, C ~ N(0, 1) / sqrt(N)          per token and state index, [Bt, L, N]
* A = -exp(U[ln 1, ln 16])          per channel and state index, [D, N], fp32
* D ~ N(0, 0.1)                     per channel, [D], fp32 (0.1 is the std)
* upstream gradients dy ~ N(0, 1)   [Bt, L, D]; dstates ~ N(0, 1) if used
* mixer around the scan (raw projections before the convolution, softplus
  and gate): xr ~ N(0, 1), dt_raw ~ N(-2, 0.5), z ~ N(0, 1) per token and
  channel; convolution taps ~ N(0, 0.5) [D, 4], convolution bias and both
  step-size biases ~ N(0, 0.1) [D]
* timestep modulation of an active block (adaptive layer norm): shift,
  scale ~ N(0, 0.3) and gate ~ N(1, 0.3) per batch row and channel, [Bt, D],
  fp32; a separate draw (`part`) per denoising step

Every tensor has its own stream id; the generator for tensor ``name`` is
``numpy.random.Generator(PCG64(SeedSequence([seed, stream_id])))``. Values are
drawn in fp32 and, for bf16 workloads, rounded to bf16 with round-to-nearest-
even. The oracle then receives the exact bf16 values widened to fp64, and the
GPU receives the bf16 bit patterns, so both sides see identical inputs.
"""

from __future__ import annotations

import numpy as np

# one stream id per tensor: the clean stream, the shared noisy tokens, the
# forward-direction and reverse-direction projections, parameters, gradients
STREAM_IDS = {
    "x_c": 0, "dt_c": 1, "B_c": 2, "C_c": 3,
    "x_n": 4,
    "dt_f": 5, "B_f": 6, "C_f": 7,
    "dt_r": 8, "B_r": 9, "C_r": 10,
    "A_f": 11, "D_f": 12, "A_r": 13, "D_r": 14,
    "dy_c": 15, "dy_n": 16, "dstates": 17, "init_state": 18,
    "shift": 19, "scale": 20, "gate": 21,
    "xr_c": 22, "xr_n": 23, "dtr_c": 24, "dtr_f": 25, "dtr_r": 26, "z_c": 27, "z_n": 28,
    "conv_w": 29, "conv_b": 30, "dt_bias_f": 31, "dt_bias_r": 32,
}

TOKEN_D = ("x_c", "dt_c", "x_n", "dt_f", "dt_r")       # [Bt, L, D]
TOKEN_N = ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r")   # [Bt, L, N]
PARAMS = ("A_f", "D_f", "A_r", "D_r")                  # fp32 always


def _rng(seed: int, name: str, part: int = 0) -> np.random.Generator:
    key = [int(seed), STREAM_IDS[name]] + ([int(part)] if part else [])
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(key)))


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round finite fp32 values to bf16 (round to nearest, ties to even);
    returns uint16 bits. (uint32 arithmetic cannot overflow for finite input.)"""
    u = np.ascontiguousarray(a, dtype=np.float32).reshape(-1).view(np.uint32)
    out = np.empty(u.shape, dtype=np.uint16)
    step = 1 << 24
    for i in range(0, u.size, step):
        v = u[i:i + step]
        out[i:i + step] = ((v + np.uint32(0x7FFF) + ((v >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)).astype(np.uint16)
    return out.reshape(np.shape(a))


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _softplus32(z: np.ndarray) -> np.ndarray:
    # log(1 + e^z), evaluated stably in fp32 (input distribution only)
    z = z.astype(np.float32)
    return (np.maximum(z, 0) + np.log1p(np.exp(-np.abs(z)))).astype(np.float32)


def draw(name: str, shape, seed: int, part: int = 0) -> np.ndarray:
    """fp32 draw for one named tensor, following the module recipe. `part`
    selects an independent draw of the same tensor (e.g. successive noisy
    blocks of a denoising loop)."""
    g = _rng(seed, name, part)
    if name in ("x_c", "x_n", "dy_c", "dy_n", "dstates", "init_state"):
        return g.standard_normal(shape, dtype=np.float32)
    if name in ("dt_c", "dt_f", "dt_r"):
        return _softplus32(g.normal(-2.0, 0.5, size=shape).astype(np.float32))
    if name in TOKEN_N:
        n = shape[-1]
        return (g.standard_normal(shape, dtype=np.float32) / np.float32(np.sqrt(n))).astype(np.float32)
    if name in ("A_f", "A_r"):
        u = g.uniform(np.log(1.0), np.log(16.0), size=shape)
        return (-np.exp(u)).astype(np.float32)
    if name in ("D_f", "D_r"):
        return g.normal(0.0, 0.1, size=shape).astype(np.float32)
    if name in ("xr_c", "xr_n", "z_c", "z_n"):
        return g.standard_normal(shape, dtype=np.float32)
    if name in ("dtr_c", "dtr_f", "dtr_r"):
        return g.normal(-2.0, 0.5, size=shape).astype(np.float32)
    if name == "conv_w":
        return g.normal(0.0, 0.5, size=shape).astype(np.float32)
    if name in ("conv_b", "dt_bias_f", "dt_bias_r"):
        return g.normal(0.0, 0.1, size=shape).astype(np.float32)
    if name in ("shift", "scale"):
        return g.normal(0.0, 0.3, size=shape).astype(np.float32)
    if name == "gate":
        return g.normal(1.0, 0.3, size=shape).astype(np.float32)
    raise KeyError(name)


class Workload:
    """One seeded problem instance.

    ``t32[name]`` holds every tensor as fp32 (already bf16-rounded for bf16
    workloads), ``f64(name)`` the same values widened to fp64 for the oracle,
    and ``dev_bits(name)`` the array handed to the GPU (uint16 bf16 bits for
    bf16 workloads, fp32 otherwise; parameters are always fp32).
    """

    def __init__(self, batch, length, block, d_inner, d_state, dtype="bf16", seed=0,
                 with_grads=True, with_dstates=False, with_init=False, parts=("clean", "noisy"), part=0):
        if dtype not in ("bf16", "f32"):
            raise ValueError(dtype)
        self.batch, self.len, self.block = int(batch), int(length), int(block)
        self.d_inner, self.d_state, self.dtype, self.seed = int(d_inner), int(d_state), dtype, int(seed)
        Bt, L, D, N = self.batch, self.len, self.d_inner, self.d_state
        nb = L // self.block if self.block > 0 else 0
        shapes = {}
        for k in TOKEN_D:
            if ("clean" in parts and k.endswith("_c")) or ("noisy" in parts and not k.endswith("_c")):
                shapes[k] = (Bt, L, D)
        for k in TOKEN_N:
            if ("clean" in parts and k.endswith("_c")) or ("noisy" in parts and not k.endswith("_c")):
                shapes[k] = (Bt, L, N)
        shapes.update({"A_f": (D, N), "A_r": (D, N), "D_f": (D,), "D_r": (D,)})
        if with_grads:
            shapes.update({"dy_c": (Bt, L, D), "dy_n": (Bt, L, D)})
        if with_dstates:
            shapes["dstates"] = (Bt, nb, D, N)
        if with_init:
            shapes["init_state"] = (Bt, D, N)
        self.t32 = {}
        for k, shp in shapes.items():
            a = draw(k, shp, self.seed, 0 if k in PARAMS else part)
            if dtype == "bf16" and k not in PARAMS and k not in ("dstates", "init_state"):
                a = bf16_bits_to_f32(f32_to_bf16_bits(a)).reshape(shp)
            self.t32[k] = a

    def f64(self, name: str) -> np.ndarray:
        return self.t32[name].astype(np.float64)

    def dev_bits(self, name: str) -> np.ndarray:
        a = self.t32[name]
        if self.dtype == "bf16" and name not in PARAMS and name not in ("dstates", "init_state"):
            return f32_to_bf16_bits(a).reshape(a.shape)
        return a

    def override(self, name: str, value) -> None:
        """Replace one tensor (already in the workload's number format)."""
        a = np.asarray(value, dtype=np.float32).reshape(self.t32[name].shape)
        if self.dtype == "bf16" and name not in PARAMS and name not in ("dstates", "init_state"):
            a = bf16_bits_to_f32(f32_to_bf16_bits(a)).reshape(a.shape)
        self.t32[name] = np.ascontiguousarray(a)


class SsdWorkload(Workload):
    """A seeded problem instance of the SSD (Mamba-2) form: x [Bt, L, H, 64],
    dt [Bt, L, H], B, C [Bt, L, N], A and D per head [H]; init_state and seeds
    [Bt, H, 64, N]. Same draws as the diagonal layer (same stream ids and value
    recipe), with these shapes; the forward-side tensors only."""

    def __init__(self, batch, length, block, heads, d_state, seed=0, with_init=False, head_dim=64, part=0,
                 with_grads=False, with_dstates=False):
        self.batch, self.len, self.block = int(batch), int(length), int(block)
        self.heads, self.head_dim, self.d_state = int(heads), int(head_dim), int(d_state)
        self.d_inner, self.dtype, self.seed = self.heads * self.head_dim, "bf16", int(seed)
        Bt, L, H, P, N = self.batch, self.len, self.heads, self.head_dim, self.d_state
        shapes = {"x_c": (Bt, L, H, P), "dt_c": (Bt, L, H), "B_c": (Bt, L, N), "C_c": (Bt, L, N),
                  "x_n": (Bt, L, H, P), "dt_f": (Bt, L, H), "B_f": (Bt, L, N), "C_f": (Bt, L, N),
                  "dt_r": (Bt, L, H), "B_r": (Bt, L, N), "C_r": (Bt, L, N),
                  "A_f": (H,), "A_r": (H,), "D_f": (H,), "D_r": (H,)}
        if with_init:
            shapes["init_state"] = (Bt, H, P, N)
        if with_grads:
            shapes.update({"dy_c": (Bt, L, H, P), "dy_n": (Bt, L, H, P)})
        if with_dstates:
            shapes["dstates"] = (Bt, L // self.block, H, P, N)
        self.t32 = {}
        for k, shp in shapes.items():
            a = draw(k, shp, self.seed, 0 if k in PARAMS else part)
            if k not in PARAMS and k not in ("init_state", "dstates"):
                a = bf16_bits_to_f32(f32_to_bf16_bits(a)).reshape(shp)
            self.t32[k] = a


MIXER_PARAMS = ("A_f", "D_f", "A_r", "D_r", "conv_w", "conv_b", "dt_bias_f", "dt_bias_r")


class MixerWorkload(Workload):
    """A seeded problem instance of the mixer around the scan: the raw inputs
    xr, dt_raw and gates z of both streams ([Bt, L, D]), B and C ([Bt, L, N]),
    the scan parameters and the convolution and step-size parameters (fp32),
    and the upstream gradients dout (drawn like dy) of both streams."""

    TOKEN = ("xr_c", "dtr_c", "z_c", "xr_n", "dtr_f", "dtr_r", "z_n")

    def __init__(self, batch, length, block, d_inner, d_state, dtype="bf16", seed=0, with_grads=True,
                 parts=("clean", "noisy"), part=0, with_init=False):
        if dtype not in ("bf16", "f32"):
            raise ValueError(dtype)
        self.batch, self.len, self.block = int(batch), int(length), int(block)
        self.d_inner, self.d_state, self.dtype, self.seed = int(d_inner), int(d_state), dtype, int(seed)
        Bt, L, D, N = self.batch, self.len, self.d_inner, self.d_state
        shapes = {}
        for k in self.TOKEN:
            if ("clean" in parts and k.endswith("_c")) or ("noisy" in parts and not k.endswith("_c")):
                shapes[k] = (Bt, L, D)
        for k in TOKEN_N:
            if ("clean" in parts and k.endswith("_c")) or ("noisy" in parts and not k.endswith("_c")):
                shapes[k] = (Bt, L, N)
        shapes.update({"A_f": (D, N), "A_r": (D, N), "D_f": (D,), "D_r": (D,), "conv_w": (D, 4), "conv_b": (D,),
                       "dt_bias_f": (D,), "dt_bias_r": (D,)})
        if with_grads:
            shapes.update({"dy_c": (Bt, L, D), "dy_n": (Bt, L, D)})
        if with_init:
            shapes["init_state"] = (Bt, D, N)
        self.t32 = {}
        for k, shp in shapes.items():
            a = draw(k, shp, self.seed, 0 if k in MIXER_PARAMS else part)
            if dtype == "bf16" and k not in MIXER_PARAMS and k != "init_state":
                a = bf16_bits_to_f32(f32_to_bf16_bits(a)).reshape(shp)
            self.t32[k] = a

    def dev_bits(self, name: str) -> np.ndarray:
        a = self.t32[name]
        if self.dtype == "bf16" and name not in MIXER_PARAMS and name != "init_state":
            return f32_to_bf16_bits(a).reshape(a.shape)
        return a
