"""GPU parity of the mixer around the scan (include/bdscan_mixer.h): the width-4
causal convolution with its cache state, softplus step size and SiLU gate,
through the C ABI, against the fp64 oracle (oracle/mixer.py) on the same
seeded inputs, forward and every gradient; the cache (SSM and convolution
states) reproduces the all-block output bit for bit."""

import numpy as np
import pytest

import parity as P
from paper_2607_02805_gb300.inputs import MixerWorkload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import to_device, to_numpy  # noqa: E402

FWD = ("xr_c", "dtr_c", "B_c", "C_c", "z_c", "xr_n", "dtr_f", "B_f", "C_f", "dtr_r", "B_r", "C_r", "z_n",
       "A_f", "D_f", "A_r", "D_r", "conv_w", "conv_b", "dt_bias_f", "dt_bias_r")
ORACLE_NAMES = {"conv_w": "w", "conv_b": "b", "dt_bias_f": "bias_f", "dt_bias_r": "bias_r"}
PER_CHANNEL_PARAMS = ("A_f", "D_f", "A_r", "D_r", "conv_w", "conv_b", "dt_bias_f", "dt_bias_r")
TOKEN_N = ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r")


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


def _dev(wl, code):
    return {k: to_device(wl.dev_bits(k), code, "cuda") for k in wl.t32}


def _run(wl, od=None, want_bwd=True):
    code = binding.BDSCAN_BF16 if wl.dtype == "bf16" else binding.BDSCAN_F32
    dims = binding.make_dims(wl.batch, wl.len, wl.block, wl.d_inner, wl.d_state, code, od)
    t = _dev(wl, code)
    out_t = torch.float32 if (wl.dtype == "f32" or od == binding.BDSCAN_F32) else torch.bfloat16
    Bt, L, D, N = wl.batch, wl.len, wl.d_inner, wl.d_state
    out_c = torch.full((Bt, L, D), float("nan"), dtype=out_t, device="cuda")
    out_n = torch.full_like(out_c, float("nan"))
    st = torch.empty((Bt, L // wl.block, D, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.bdscan_mixer_forward_workspace_size(dims), dtype=torch.uint8, device="cuda")
    binding.mixer_forward(dims, t, out_c, out_n, st, ws)
    g = None
    if want_bwd:
        g = {}
        for k, v in t.items():
            if k in ("dy_c", "dy_n"):
                continue
            g[k] = torch.full(v.shape, float("nan"), dtype=torch.float32 if k in PER_CHANNEL_PARAMS else out_t,
                              device="cuda")
        wsb = torch.empty(binding.bdscan_mixer_backward_workspace_size(dims), dtype=torch.uint8, device="cuda")
        binding.mixer_backward(dims, t, t["dy_c"], t["dy_n"], None, g, wsb)
    torch.cuda.synchronize()
    return dims, t, out_c, out_n, st, g, (P.BF16_U if out_t == torch.bfloat16 else 0.0)


def _oracle_inputs(wl, sub=None):
    d = {}
    for k in FWD + ("dy_c", "dy_n"):
        if k not in wl.t32:
            continue
        a = wl.f64(k)
        if sub is not None:
            if k in PER_CHANNEL_PARAMS:
                a = a[sub]
            elif k not in TOKEN_N:
                a = a[:, :, sub]
        d[ORACLE_NAMES.get(k, k)] = np.ascontiguousarray(a)
    return d


def _check(wl, out_c, out_n, st, g, u, sub=None, sums=True):
    from oracle import mixer
    d = _oracle_inputs(wl, sub)
    args = [d[ORACLE_NAMES.get(k, k)] for k in FWD]
    oc, on, ost = mixer.forward(wl.block, *args)
    pick = (lambda a: a) if sub is None else (lambda a: a[:, :, sub])
    P.assert_close("out_c", pick(to_numpy(out_c)), oc, P.FWD_TOL, u)
    P.assert_close("out_n", pick(to_numpy(out_n)), on, P.FWD_TOL, u)
    P.assert_close("states", pick(to_numpy(st)), ost, P.FWD_TOL)
    if g is None:
        return
    og = mixer.backward(wl.block, *args, d["dy_c"], d["dy_n"])
    for k in FWD:
        if k in TOKEN_N and not sums:
            continue
        gpu = to_numpy(g[k])
        if sub is not None:
            gpu = gpu[sub] if k in PER_CHANNEL_PARAMS else (gpu if k in TOKEN_N else gpu[:, :, sub])
        P.assert_close("d" + k, gpu, og[ORACLE_NAMES.get(k, k)], P.GRAD_TOL, 0.0 if k in PER_CHANNEL_PARAMS else u)


@pytest.mark.parametrize("Bt,L,Bs,D,N,dt,od,seed", [
    (2, 256, 16, 136, 16, "bf16", None, 61),                # ragged channel group, 2 chunks
    (1, 96, 4, 64, 8, "f32", None, 62),                     # short blocks
    (2, 48, 2, 40, 16, "f32", None, 63),                    # convolution windows spanning several blocks
    (1, 256, 32, 128, 16, "bf16", binding.BDSCAN_F32, 64),  # 2 backward segments per block
    (1, 64, 1, 32, 16, "bf16", None, 65),                   # block size 1
])
def test_mixer_forward_backward_matches_oracle(Bt, L, Bs, D, N, dt, od, seed):
    wl = MixerWorkload(Bt, L, Bs, D, N, dtype=dt, seed=seed)
    _, _, out_c, out_n, st, g, u = _run(wl, od)
    _check(wl, out_c, out_n, st, g, u)


def test_mixer_87m_layer_sampled_channels():
    """The 87M-scale layer's geometry (d_inner 1536, d_state 16, block 16) at
    batch 2 x 2048 tokens: per-channel outputs and gradients on a channel
    sample; the channel sums dB, dC checked on the whole problem's channels
    is left to the small cases above."""
    wl = MixerWorkload(2, 2048, 16, 1536, 16, dtype="bf16", seed=66)
    _, _, out_c, out_n, st, g, u = _run(wl)
    sub = [0, 1, 127, 128, 700, 1535]
    _check(wl, out_c, out_n, st, g, u, sub=sub, sums=False)


@pytest.mark.parametrize("Bs", [2, 16, 32])
def test_mixer_cache_with_convolution_state_is_bit_exact(Bs):
    """Cache build over the prefix (SSM and convolution states), then the
    cached active block, equals the all-block forward's last noisy block."""
    Bt, L, D, N = 2, 8 * Bs if Bs > 2 else 32, 136, 16
    wl = MixerWorkload(Bt, L, Bs, D, N, dtype="bf16", seed=67, with_grads=False)
    dims, t, out_c, out_n, st, _, _ = _run(wl, want_bwd=False)
    pre = {k: (v[:, : L - Bs].contiguous() if v.dim() == 3 else v) for k, v in t.items()}
    dp = binding.make_dims(Bt, L - Bs, Bs, D, N, binding.BDSCAN_BF16)
    ws = torch.empty(binding.bdscan_mixer_boundary_states_workspace_size(dp), dtype=torch.uint8, device="cuda")
    sts = torch.empty((Bt, (L - Bs) // Bs, D, N), dtype=torch.float32, device="cuda")
    cst = torch.empty((Bt, (L - Bs) // Bs, 3, D), dtype=torch.float32, device="cuda")
    yc = torch.empty((Bt, L - Bs, D), dtype=torch.bfloat16, device="cuda")
    binding.mixer_boundary_states(dp, pre, None, None, yc, sts, cst, 1, ws)
    fin = torch.empty((Bt, 1, D, N), dtype=torch.float32, device="cuda")
    cfin = torch.empty((Bt, 1, 3, D), dtype=torch.float32, device="cuda")
    binding.mixer_boundary_states(dp, pre, None, None, None, fin, cfin, 0, ws)
    blk = {k: (v[:, L - Bs:].contiguous() if v.dim() == 3 else v) for k, v in t.items()}
    da = binding.make_dims(Bt, Bs, Bs, D, N, binding.BDSCAN_BF16)
    wsa = torch.empty(binding.bdscan_mixer_active_block_workspace_size(da), dtype=torch.uint8, device="cuda")
    ya = torch.full((Bt, Bs, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    binding.mixer_active_block(da, fin[:, 0].contiguous(), cfin[:, 0].contiguous(), blk, ya, wsa)
    torch.cuda.synchronize()
    assert torch.equal(sts, st[:, :-1])
    assert torch.equal(fin[:, 0], st[:, -2])
    assert torch.equal(yc, out_c[:, : L - Bs])
    assert torch.equal(cfin[:, 0], cst[:, -1])
    # the convolution state is the clean raw input of the prefix's last 3 tokens
    assert torch.equal(cfin[:, 0], t["xr_c"][:, L - Bs - 3: L - Bs].float())
    assert torch.equal(ya, out_n[:, L - Bs:])
    # and the cached step against the oracle
    from oracle import mixer
    d = _oracle_inputs(wl)
    s64, c64 = mixer.boundary_states(Bs, d["xr_c"][:, : L - Bs], d["dtr_c"][:, : L - Bs], d["B_c"][:, : L - Bs],
                                     d["C_c"][:, : L - Bs], d["A_f"], d["D_f"], d["w"], d["b"], d["bias_f"],
                                     emit_all=False)
    P.assert_close("cached state", to_numpy(fin), s64, P.FWD_TOL)
    assert np.array_equal(to_numpy(cfin), c64)
    sl = slice(L - Bs, L)
    oy = mixer.active_block(s64[:, 0], c64[:, 0], d["xr_n"][:, sl], d["dtr_f"][:, sl], d["B_f"][:, sl],
                            d["C_f"][:, sl], d["dtr_r"][:, sl], d["B_r"][:, sl], d["C_r"][:, sl], d["z_n"][:, sl],
                            d["A_f"], d["D_f"], d["A_r"], d["D_r"], d["w"], d["b"], d["bias_f"], d["bias_r"])
    P.assert_close("cached active block", to_numpy(ya), oy, P.FWD_TOL, P.BF16_U)


def test_mixer_cache_append_from_an_initial_state():
    """Appending: the second half of a prefix continued from the first half's
    SSM and convolution states equals one cache build (oracle check)."""
    Bt, L, Bs, D, N = 1, 512, 16, 64, 16
    wl = MixerWorkload(Bt, L, Bs, D, N, dtype="bf16", seed=68, with_grads=False, parts=("clean",))
    t = _dev(wl, binding.BDSCAN_BF16)
    h = L // 2

    def build(tt, length, init=None, cinit=None):
        dd = binding.make_dims(Bt, length, Bs, D, N, binding.BDSCAN_BF16)
        ws = torch.empty(binding.bdscan_mixer_boundary_states_workspace_size(dd), dtype=torch.uint8, device="cuda")
        s = torch.empty((Bt, 1, D, N), dtype=torch.float32, device="cuda")
        c = torch.empty((Bt, 1, 3, D), dtype=torch.float32, device="cuda")
        binding.mixer_boundary_states(dd, tt, init, cinit, None, s, c, 0, ws)
        return s, c

    a_s, a_c = build({k: (v[:, :h].contiguous() if v.dim() == 3 else v) for k, v in t.items()}, h)
    b_s, b_c = build({k: (v[:, h:].contiguous() if v.dim() == 3 else v) for k, v in t.items()}, L - h,
                     a_s[:, 0].contiguous(), a_c[:, 0].contiguous())
    f_s, f_c = build(t, L)
    torch.cuda.synchronize()
    assert torch.equal(b_c, f_c)
    from oracle import mixer
    d = {k: wl.f64(k) for k in wl.t32}
    s64, _ = mixer.boundary_states(Bs, d["xr_c"], d["dtr_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"], d["conv_w"],
                                   d["conv_b"], d["dt_bias_f"], emit_all=False)
    P.assert_close("appended state", to_numpy(b_s), s64, P.FWD_TOL)
    P.assert_close("one-build state", to_numpy(f_s), s64, P.FWD_TOL)
