"""bdscan_boundary_states_noalloc: the cache build for callers that may not
allocate device memory (for example a plugin running inside another engine's
pre-planned memory, or a serving loop that cannot afford a synchronising
cudaMalloc). It keeps its scratch in a static device array of the library, so
it is checked here against bdscan_boundary_states, which takes a caller
workspace, through the C ABI. Two different problems run back to back,
because every call shares the same static array and must not be affected by
what the previous call left in it.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.
"""

import numpy as np
import pytest

import parity as P
from paper_2607_02805_gb300.inputs import Workload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import to_device, to_numpy  # noqa: E402


def _problem(Bt, L, Bs, D, N, seed, with_init):
    wl = Workload(Bt, L, Bs, D, N, dtype="bf16", seed=seed, with_grads=False, with_init=with_init,
                  parts=("clean",))
    dims = binding.make_dims(Bt, L, Bs, D, N, binding.BDSCAN_BF16)
    t = {k: to_device(wl.dev_bits(k), binding.BDSCAN_BF16, "cuda") for k in wl.t32}
    clean = binding.bdscan_clean(t["x_c"].data_ptr(), t["dt_c"].data_ptr(), t["B_c"].data_ptr(),
                                 t["C_c"].data_ptr())
    return wl, dims, t, clean


def _outputs(wl, t, emit_all, want_y):
    Bt, L, Bs, D, N = wl.batch, wl.len, wl.block, wl.d_inner, wl.d_state
    st = torch.full((Bt, (L // Bs) if emit_all else 1, D, N), float("nan"), dtype=torch.float32, device="cuda")
    y = torch.full((Bt, L, D), float("nan"), dtype=torch.bfloat16, device="cuda") if want_y else None
    return st, y


def _ptr(x):
    return None if x is None else x.data_ptr()


def _run_both(Bt, L, Bs, D, N, seed, emit_all, want_y, with_init):
    wl, dims, t, clean = _problem(Bt, L, Bs, D, N, seed, with_init)
    init = t.get("init_state")
    stream = torch.cuda.current_stream().cuda_stream
    # existing entry point, with a caller workspace
    st_ws, y_ws = _outputs(wl, t, emit_all, want_y)
    nbytes = binding.bdscan_boundary_states_workspace_size(dims, emit_all)
    ws = torch.empty((nbytes + 3) // 4, dtype=torch.float32, device="cuda")
    rc = binding.bdscan_boundary_states(dims, clean, t["A_f"].data_ptr(), t["D_f"].data_ptr(), _ptr(init),
                                        _ptr(y_ws), st_ws.data_ptr(), emit_all, ws.data_ptr(), nbytes, stream)
    assert rc == binding.BDSCAN_OK, binding.bdscan_last_error()
    launches_ws = binding.bdscan_last_launch_count()
    # the entry point without a workspace
    st_na, y_na = _outputs(wl, t, emit_all, want_y)
    rc = binding.bdscan_boundary_states_noalloc(dims, clean, t["A_f"].data_ptr(), t["D_f"].data_ptr(), _ptr(init),
                                                _ptr(y_na), st_na.data_ptr(), emit_all, stream)
    assert rc == binding.BDSCAN_OK, binding.bdscan_last_error()
    # the same kernels, counted the same way by the library's launch counter
    assert binding.bdscan_last_launch_count() == launches_ws
    torch.cuda.synchronize()
    # Both paths run the same kernels on the same inputs, so the results are
    # the same bits. The tolerance check runs first only to report the size
    # of a difference, should there be one.
    P.assert_close("states", to_numpy(st_na), to_numpy(st_ws), P.FWD_TOL)
    assert torch.equal(st_na, st_ws)
    if want_y:
        P.assert_close("y_c", to_numpy(y_na), to_numpy(y_ws), P.FWD_TOL, P.BF16_U)
        assert torch.equal(y_na, y_ws)


def test_noalloc_matches_workspace_entry_point_two_calls_in_a_row():
    # first call: every block-end state and the clean outputs, several full chunks
    _run_both(2, 1024, 16, 256, 16, seed=1, emit_all=True, want_y=True, with_init=False)
    # second call, a different problem: final state only, continued from an
    # initial state, ragged last chunk (it rescans that chunk from scratch data)
    _run_both(1, 400, 16, 136, 8, seed=2, emit_all=False, want_y=False, with_init=True)
    # third call: final state only over whole chunks (512 tokens at block 16
    # are four 128-token chunks), so the final state is copied out of the
    # scratch row by row with the chunk-slot pitch
    assert 512 % binding.bdscan_chunk_tokens(16) == 0
    _run_both(2, 512, 16, 136, 16, seed=3, emit_all=False, want_y=False, with_init=True)


def test_noalloc_rejects_problems_larger_than_its_scratch():
    # a 65,536-token prefix at d_inner 2048 needs about 67 MB of chunk states
    dims = binding.make_dims(1, 65536, 32, 2048, 16, binding.BDSCAN_BF16)
    need = binding.bdscan_boundary_states_workspace_size(dims, 0)
    assert need > binding.BDSCAN_NOALLOC_SCRATCH_BYTES
    fake = 1 << 20  # aligned, never dereferenced: the size check runs before any GPU work
    clean = binding.bdscan_clean(fake, fake, fake, fake)
    rc = binding.bdscan_boundary_states_noalloc(dims, clean, fake, fake, None, None, fake, 0, None)
    assert rc == binding.BDSCAN_ERR_UNSUPPORTED
    msg = binding.bdscan_last_error()
    assert "static scratch" in msg and str(need) in msg
