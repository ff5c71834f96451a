"""The debug build (BDSCAN_DEBUG=1) on the GPU: its device status words and
BDSCAN_ERR_DEVICE, without faulting anything. A clean call returns 0 with
outputs bit-identical to the release build's; a NaN input is reported as a
non-finite cached state; and with the extents shortened by a slack the
kernels' extent checks fail on in-range accesses, the flagged CTAs skip their
work, and the call returns BDSCAN_ERR_DEVICE naming the kernel. Every check
depends on the block index and the sizes only, so no access is ever made out
of range."""

import numpy as np
import pytest

from paper_2607_02805_gb300.inputs import SsdWorkload, Workload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import Layer, to_device  # noqa: E402


@pytest.fixture
def debug_build():
    binding.use_debug_build(True)
    assert binding.bdscan_debug_build() == 1
    try:
        yield
    finally:
        binding.bdscan_debug_set_slack(0)
        binding.use_debug_build(False)


def _diag(wl, nan_at=None):
    lay = Layer(wl, device="cuda")
    if nan_at is not None:
        lay.t["x_c"][nan_at] = float("nan")
    return lay


def _outputs(lay):
    out = {"y_c": lay.y_c, "y_n": lay.y_n, "states": lay.states}
    out.update({"d" + k: v for k, v in lay.g.items()})
    return {k: v.clone() for k, v in out.items()}


def _run_diag(wl, nan_at=None):
    lay = _diag(wl, nan_at)
    lay.forward()
    lay.backward(use_dstates=False)
    torch.cuda.synchronize()
    return lay


WL = dict(batch=2, length=512, block=16, d_inner=256, d_state=16)


def _wl():
    return Workload(WL["batch"], WL["length"], WL["block"], WL["d_inner"], WL["d_state"], dtype="bf16", seed=5,
                    with_grads=True)


def test_debug_build_matches_release_bit_for_bit(debug_build):
    binding.use_debug_build(False)
    ref = _outputs(_run_diag(_wl()))
    binding.use_debug_build(True)
    got = _outputs(_run_diag(_wl()))
    for k in ref:
        assert torch.equal(ref[k], got[k]), k


def test_debug_build_reports_a_non_finite_cached_state(debug_build):
    with pytest.raises(binding.BdscanError) as e:
        _run_diag(_wl(), nan_at=(0, 5, 3))
    assert e.value.code == binding.BDSCAN_ERR_DEVICE
    assert "non-finite" in str(e.value) and "k_chunk_carry" in str(e.value)
    # the status word was cleared: a clean call succeeds again
    _run_diag(_wl())


def test_debug_build_extent_checks_skip_the_flagged_ctas(debug_build):
    binding.use_debug_build(False)
    ref = _outputs(_run_diag(_wl()))
    binding.use_debug_build(True)
    assert binding.bdscan_debug_set_slack(1) == 0
    lay = _diag(_wl())
    with pytest.raises(binding.BdscanError) as e:
        lay.forward()
    assert e.value.code == binding.BDSCAN_ERR_DEVICE
    msg = str(e.value)
    assert "outside the extent" in msg and "(the CTA skipped its work)" in msg
    assert any(k in msg for k in ("k_chunk_local", "k_chunk_carry", "k_block_scan")), msg
    # exact extents again: the same call succeeds and matches the release build
    assert binding.bdscan_debug_set_slack(0) == 0
    got = _outputs(_run_diag(_wl()))
    for k in ref:
        assert torch.equal(ref[k], got[k]), k


def _ssd(wl):
    names = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r", "D_r")
    params = ("A_f", "D_f", "A_r", "D_r")
    t = {k: to_device(wl.dev_bits(k), binding.BDSCAN_F32 if k in params else binding.BDSCAN_BF16, "cuda")
         for k in wl.t32}
    Bt, L, Bs, H, N = wl.batch, wl.len, wl.block, wl.heads, wl.d_state
    d = binding.make_ssd_dims(Bt, L, Bs, H, N)
    y_c = torch.empty((Bt, L, H, 64), dtype=torch.bfloat16, device="cuda")
    y_n = torch.empty_like(y_c)
    st = torch.empty((Bt, L // Bs, H, 64, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.bdscan_ssd_forward_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_forward(d, t, y_c, y_n, st, ws)
    g = {k: torch.empty(t[k].shape, dtype=torch.float32 if k in params else torch.bfloat16, device="cuda")
         for k in names}
    wsb = torch.empty(binding.bdscan_ssd_backward_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_backward(d, t, st, t["dy_c"], t["dy_n"], None, g, wsb)
    torch.cuda.synchronize()
    out = {"y_c": y_c, "y_n": y_n, "states": st}
    out.update({"d" + k: v for k, v in g.items()})
    return {k: v.clone() for k, v in out.items()}


def test_debug_build_ssd_form(debug_build):
    wl = SsdWorkload(1, 512, 256, 3, 128, seed=9, with_grads=True)
    binding.use_debug_build(False)
    ref = _ssd(wl)
    binding.use_debug_build(True)
    got = _ssd(wl)
    for k in ref:
        assert torch.equal(ref[k], got[k]), k
    assert binding.bdscan_debug_set_slack(1) == 0
    with pytest.raises(binding.BdscanError) as e:
        _ssd(wl)
    assert e.value.code == binding.BDSCAN_ERR_DEVICE and "k_ssd_" in str(e.value)
    assert np.isfinite(ref["states"].cpu().numpy()).all()
