"""The cached denoising loop replayed as one CUDA graph (the paper's inference
protocol, Appendix B: fixed-shape block steps captured once and replayed).

For both forms of the layer, the cache is built over a clean prefix, then 16
active-block calls read the same cached state. They are captured in one CUDA
graph and replayed. Each replayed output must equal, bit for bit, the same
call made outside a graph. It must also match the fp64 oracle. Replays run
twice with the outputs cleared in between: a graph re-runs its kernels and
does not reuse a result.
"""

import pytest

import parity as P
from paper_2607_02805_gb300.inputs import SsdWorkload, Workload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import to_device, to_numpy  # noqa: E402

CALLS = 16


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


def _replay_and_compare(call, outs):
    """Runs `call(j, stream)` for every j outside a graph, then captures all
    calls in one graph on a side stream and replays it twice; returns the
    eager outputs and checks the replays against them bit for bit."""
    stream = torch.cuda.current_stream()
    for j in range(CALLS):
        call(j, stream)
    torch.cuda.synchronize()
    eager = [o.clone() for o in outs]
    for o in outs:
        o.fill_(float("nan"))
    side = torch.cuda.Stream()
    side.wait_stream(stream)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        for j in range(CALLS):
            call(j, side)
    torch.cuda.synchronize()
    for rep in range(2):
        for o in outs:
            o.fill_(float("nan"))
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        for j in range(CALLS):
            assert torch.equal(outs[j], eager[j]), f"replay {rep}, call {j}"
    return eager


def test_diagonal_active_block_loop_in_a_graph():
    """d_inner 256, d_state 16, block 16, bf16; a 4,096-token prefix."""
    Bt, L, Bs, D, N, seed = 2, 4096, 16, 256, 16, 41
    code = binding.BDSCAN_BF16
    wl = Workload(Bt, L, Bs, D, N, dtype="bf16", seed=seed, with_grads=False, parts=("clean",))
    t = {k: to_device(wl.dev_bits(k), code, "cuda") for k in wl.t32}
    dims = binding.make_dims(Bt, L, Bs, D, N, code)
    fin = torch.empty((Bt, 1, D, N), dtype=torch.float32, device="cuda")
    ws = torch.empty((binding.bdscan_boundary_states_workspace_size(dims, 0) + 3) // 4, dtype=torch.float32,
                     device="cuda")
    binding.boundary_states(dims, t, None, None, fin, 0, ws)
    seed_state = fin[:, 0].contiguous()
    blocks = [Workload(Bt, Bs, Bs, D, N, dtype="bf16", seed=seed, with_grads=False, parts=("noisy",), part=j + 1)
              for j in range(CALLS)]
    tb = [{k: to_device(b.dev_bits(k), code, "cuda") for k in b.t32} for b in blocks]
    outs = [torch.empty((Bt, Bs, D), dtype=torch.bfloat16, device="cuda") for _ in range(CALLS)]
    bdims = binding.make_dims(Bt, Bs, Bs, D, N, code)

    def call(j, s):
        binding.active_block(bdims, seed_state, tb[j], outs[j], s)

    eager = _replay_and_compare(call, outs)
    # the cache is read only: the seed is unchanged after 3 x 16 calls
    torch.cuda.synchronize()
    assert torch.equal(seed_state, fin[:, 0])
    # against the oracle: the cache from the oracle's own prefix scan
    import oracle
    d = P.slice_channels(wl, None)
    ofin, _ = oracle.boundary_states(Bs, d["x_c"], d["dt_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"], emit_all=False)
    P.assert_close("cached state", to_numpy(fin), ofin, P.FWD_TOL)
    for j, b in enumerate(blocks):
        db = P.slice_channels(b, None)
        oy = oracle.active_block(ofin[:, 0], db["x_n"], db["dt_f"], db["B_f"], db["C_f"], db["dt_r"], db["B_r"],
                                 db["C_r"], db["A_f"], db["D_f"], db["A_r"], db["D_r"])
        P.assert_close(f"active block {j}", to_numpy(eager[j]), oy, P.FWD_TOL, P.BF16_U)


def test_ssd_active_block_loop_in_a_graph():
    """SSD form: 4 heads of 64, state 128, block 256; a 2,048-token prefix."""
    Bt, L, Bs, H, N, seed = 1, 2048, 256, 4, 128, 42
    wl = SsdWorkload(Bt, L, Bs, H, N, seed=seed)

    def dev(w):
        return {k: to_device(w.dev_bits(k), binding.BDSCAN_F32 if k in P.PARAMS else binding.BDSCAN_BF16, "cuda")
                for k in w.t32}

    t = dev(wl)
    d = binding.make_ssd_dims(Bt, L, Bs, H, N)
    fin = torch.empty((Bt, 1, H, 64, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.bdscan_ssd_boundary_states_workspace_size(d, 0), dtype=torch.uint8, device="cuda")
    binding.ssd_boundary_states(d, t, None, None, fin, 0, ws)
    seed_state = fin[:, 0].contiguous()
    blocks = [SsdWorkload(Bt, Bs, Bs, H, N, seed=seed, part=j + 1) for j in range(CALLS)]
    tb = [dev(b) for b in blocks]
    outs = [torch.empty((Bt, Bs, H, 64), dtype=torch.bfloat16, device="cuda") for _ in range(CALLS)]
    da = binding.make_ssd_dims(Bt, Bs, Bs, H, N)

    def call(j, s):
        binding.ssd_active_block(da, seed_state, tb[j], outs[j], s)

    eager = _replay_and_compare(call, outs)
    assert binding.bdscan_ssd_wait_flag(1) == 0
    assert torch.equal(seed_state, fin[:, 0])
    from oracle import ssd
    o = ssd.boundary_states(Bs, *[wl.f64(k) for k in ("x_c", "dt_c", "B_c", "C_c", "A_f", "D_f")], emit_all=False)
    ofin = o[0]
    P.assert_close("cached state", to_numpy(fin), ofin, P.FWD_TOL)
    for j, b in enumerate(blocks):
        args = [b.f64(k) for k in ("x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r", "D_r")]
        oy = ssd.active_block(ofin[:, 0], *args)
        P.assert_close(f"ssd active block {j}", to_numpy(eager[j]), oy, P.FWD_TOL, P.BF16_U)
