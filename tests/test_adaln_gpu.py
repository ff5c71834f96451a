"""The timestep-modulated active block on the GPU (Appendix E, eq.
cacheable-adaln): adaptive layer norm on the active block only, through the C
ABI, against the fp64 oracle (oracle/adaln.py) on the same seeded inputs.

A denoising trajectory of 16 steps reuses one cached prefix state. Every step
has its own shift, scale and gate (its own timestep). The loop is captured in
one CUDA graph; the replay equals the eager calls bit for bit, and the cache
stays unchanged.
"""

import pytest

import parity as P
from paper_2607_02805_gb300.inputs import Workload, draw

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import to_device, to_numpy  # noqa: E402

EPS = 1e-5
NOISY = ("x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r", "D_r")


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


def _mod(Bt, D, seed, step):
    return {k: draw(k, (Bt, D), seed, step) for k in ("shift", "scale", "gate")}


def _oracle(seed_state, blk, mod):
    from oracle import adaln
    d = P.slice_channels(blk, None)
    return adaln.active_block_adaln(seed_state, *[d[k] for k in NOISY], mod["shift"], mod["scale"], mod["gate"], EPS)


def _setup(Bt, L, Bs, D, N, dtype, seed):
    code = binding.BDSCAN_BF16 if dtype == "bf16" else binding.BDSCAN_F32
    pre = Workload(Bt, L, Bs, D, N, dtype=dtype, seed=seed, with_grads=False, parts=("clean",))
    t = {k: to_device(pre.dev_bits(k), code, "cuda") for k in pre.t32}
    dims = binding.make_dims(Bt, L, Bs, D, N, code)
    fin = torch.empty((Bt, 1, D, N), dtype=torch.float32, device="cuda")
    ws = torch.empty((binding.bdscan_boundary_states_workspace_size(dims, 0) + 3) // 4, dtype=torch.float32,
                     device="cuda")
    binding.boundary_states(dims, t, None, None, fin, 0, ws)
    torch.cuda.synchronize()
    return code, fin[:, 0].contiguous()


@pytest.mark.parametrize("Bt,L,Bs,D,N,dtype,seed", [
    (2, 512, 16, 136, 16, "bf16", 51),   # ragged channel group
    (1, 256, 32, 256, 8, "f32", 52),
    (2, 1024, 64, 64, 16, "bf16", 53),
])
def test_active_block_adaln_matches_oracle(Bt, L, Bs, D, N, dtype, seed):
    code, seed_state = _setup(Bt, L, Bs, D, N, dtype, seed)
    blk = Workload(Bt, Bs, Bs, D, N, dtype=dtype, seed=seed, with_grads=False, parts=("noisy",), part=1)
    tb = {k: to_device(blk.dev_bits(k), code, "cuda") for k in blk.t32}
    mod = _mod(Bt, D, seed, 1)
    md = {k: torch.from_numpy(v).cuda() for k, v in mod.items()}
    bdims = binding.make_dims(Bt, Bs, Bs, D, N, code)
    ws = torch.empty((binding.bdscan_active_block_adaln_workspace_size(bdims) + 3) // 4, dtype=torch.float32,
                     device="cuda")
    out = torch.full((Bt, Bs, D), float("nan"), dtype=tb["x_n"].dtype, device="cuda")
    binding.active_block_adaln(bdims, seed_state, tb, md["shift"], md["scale"], md["gate"], EPS, out, ws)
    torch.cuda.synchronize()
    o = _oracle(to_numpy(seed_state), blk, mod)
    P.assert_close("adaln out", to_numpy(out), o, P.FWD_TOL, P.BF16_U if dtype == "bf16" else 0.0)


def test_adaln_denoising_loop_in_a_graph_keeps_the_cache():
    """16 denoising steps of one block (a fresh timestep modulation and a fresh
    noisy draw per step) from one cached state, replayed as a CUDA graph."""
    Bt, L, Bs, D, N, seed, steps = 1, 4096, 32, 512, 16, 54, 16
    code, seed_state = _setup(Bt, L, Bs, D, N, "bf16", seed)
    keep = seed_state.clone()
    blocks = [Workload(Bt, Bs, Bs, D, N, dtype="bf16", seed=seed, with_grads=False, parts=("noisy",), part=j + 1)
              for j in range(steps)]
    tb = [{k: to_device(b.dev_bits(k), code, "cuda") for k in b.t32} for b in blocks]
    mods = [_mod(Bt, D, seed, j + 1) for j in range(steps)]
    md = [{k: torch.from_numpy(v).cuda() for k, v in m.items()} for m in mods]
    bdims = binding.make_dims(Bt, Bs, Bs, D, N, code)
    ws = torch.empty((binding.bdscan_active_block_adaln_workspace_size(bdims) + 3) // 4, dtype=torch.float32,
                     device="cuda")
    outs = [torch.empty((Bt, Bs, D), dtype=torch.bfloat16, device="cuda") for _ in range(steps)]

    def call(j, s):
        binding.active_block_adaln(bdims, seed_state, tb[j], md[j]["shift"], md[j]["scale"], md[j]["gate"], EPS,
                                   outs[j], ws, s)

    stream = torch.cuda.current_stream()
    for j in range(steps):
        call(j, stream)
    torch.cuda.synchronize()
    eager = [o.clone() for o in outs]
    side = torch.cuda.Stream()
    side.wait_stream(stream)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        for j in range(steps):
            call(j, side)
    torch.cuda.synchronize()
    for o in outs:
        o.fill_(float("nan"))
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    for j in range(steps):
        assert torch.equal(outs[j], eager[j]), j
    # the prefix cache carries no timestep: untouched by 32 modulated steps
    assert torch.equal(seed_state, keep)
    for j, b in enumerate(blocks):
        o = _oracle(to_numpy(keep), b, mods[j])
        P.assert_close(f"adaln step {j}", to_numpy(eager[j]), o, P.FWD_TOL, P.BF16_U)
