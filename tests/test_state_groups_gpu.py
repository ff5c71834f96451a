"""d_state above 16 (or not 8 or 16) in the diagonal form: the scans run per
group of 16 states (the last one 8 or 16, zero-padded) and the groups'
outputs are added. GPU parity against the fp64 oracle, which takes any N,
element by element; and the cache paths stay bit-exact against the all-block
output."""

import pytest

import parity as P
from paper_2607_02805_gb300.inputs import Workload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import Layer  # noqa: E402
from test_parity_gpu import _active, _boundary, _check_forward, _check_grads, _sub_workload  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


GROUPED = [  # (Bt, L, Bs, D, N, dtype, out_dtype, seed): N = 4 (one padded group of 8), 12 (padded 16),
    (1, 256, 16, 64, 4, "f32", None, 81),            # 24 (16 + 8), 32, 48, 64 (four groups)
    (2, 256, 16, 72, 12, "bf16", None, 82),
    (1, 384, 32, 64, 24, "bf16", binding.BDSCAN_F32, 83),
    (2, 256, 8, 128, 32, "bf16", None, 84),
    (1, 256, 16, 64, 48, "f32", None, 85),
    (2, 512, 16, 96, 64, "bf16", None, 86),
]


@pytest.mark.parametrize("Bt,L,Bs,D,N,dt,od,seed", GROUPED)
def test_grouped_forward_backward_parity(Bt, L, Bs, D, N, dt, od, seed):
    wl = Workload(Bt, L, Bs, D, N, dtype=dt, seed=seed, with_grads=True)
    lay = Layer(wl, out_dtype=od)
    lay.forward()
    lay.backward(use_dstates=False)
    torch.cuda.synchronize()
    y_c, y_n, st = P.oracle_forward(wl)
    _check_forward(lay, y_c, y_n, st)
    g = P.oracle_backward(wl, st)
    _check_grads(lay, g)


def test_grouped_external_state_gradient_and_no_clean_output_gradient():
    wl = Workload(2, 256, 16, 64, 40, dtype="bf16", seed=87, with_grads=True, with_dstates=True)
    lay = Layer(wl, out_dtype=binding.BDSCAN_F32)
    lay.forward()
    lay.backward(use_dy_c=False, use_dstates=True)
    torch.cuda.synchronize()
    _, _, st = P.oracle_forward(wl)
    g = P.oracle_backward(wl, st, use_dy_c=False, use_dstates=True)
    _check_grads(lay, g)


@pytest.mark.parametrize("N", [64, 20])
def test_grouped_cache_reuse_is_bit_exact(N):
    """Cache build over the prefix and the cached active block reproduce the
    all-block forward bit for bit with state groups (same groups, same order
    of the additions)."""
    L, Bs = 256, 16
    wl = Workload(2, L, Bs, 64, N, dtype="bf16", seed=88, with_grads=False)
    lay = Layer(wl)
    lay.forward()
    pre = _sub_workload(wl, 0, L - Bs)
    fin, _ = _boundary(pre, emit_all=False)
    allst, y_pre = _boundary(pre, emit_all=True, want_y=True)
    blk = _sub_workload(wl, L - Bs, L)
    y = _active(blk, fin[:, 0])
    torch.cuda.synchronize()
    assert torch.equal(allst, lay.states[:, :-1])
    assert torch.equal(fin[:, 0], lay.states[:, -2])
    assert torch.equal(y_pre, lay.y_c[:, : L - Bs])
    assert torch.equal(y, lay.y_n[:, L - Bs:])


def test_grouped_backward_is_deterministic():
    wl = Workload(1, 256, 16, 64, 48, dtype="bf16", seed=89, with_grads=True)
    lay = Layer(wl)
    lay.forward()
    lay.backward(use_dstates=False)
    first = {k: v.clone() for k, v in lay.g.items()}
    lay.backward(use_dstates=False)
    torch.cuda.synchronize()
    for k in first:
        assert torch.equal(first[k], lay.g[k]), k
