"""The C ABI on the host: the library builds and loads, exports every function
include/bdscan.h declares, and rejects bad arguments before touching a GPU."""

import ctypes
import os
import re

import pytest

from paper_2607_02805_gb300 import binding

INCLUDE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
HEADERS = [os.path.join(INCLUDE, h) for h in ("bdscan.h", "bdscan_ssd.h", "bdscan_mixer.h")]


def header_functions():
    names = set()
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names.update(re.findall(r"\b(bdscan_\w+)\s*\(", text))
    return sorted(names)


def test_library_exports_every_declared_function():
    lib = binding.load()
    names = header_functions()
    assert len(names) >= 10
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(n for n, _, _ in binding.SIGNATURES) == names


def test_version_and_chunking():
    assert binding.bdscan_version() >= 100
    # chunks are whole blocks, about 128 tokens, and depend on the block size only
    assert binding.bdscan_chunk_tokens(16) == 128
    assert binding.bdscan_chunk_tokens(4) == 128
    assert binding.bdscan_chunk_tokens(48) == 96
    assert binding.bdscan_chunk_tokens(5) == 125
    assert binding.bdscan_chunk_tokens(256) == 256
    assert binding.bdscan_chunk_tokens(0) == 0


def _dims(**kw):
    base = dict(batch=2, length=64, block=16, d_inner=32, d_state=16, dtype=binding.BDSCAN_BF16)
    base.update(kw)
    return binding.make_dims(base["batch"], base["length"], base["block"], base["d_inner"], base["d_state"],
                             base["dtype"], base.get("out_dtype"))


def test_workspace_sizes():
    d = _dims(batch=8, length=2048, block=16, d_inner=1536, d_state=16)
    nc = 2048 // 128
    al = lambda x: (x + 255) // 256 * 256
    assert binding.bdscan_forward_workspace_size(d) == al(8 * (nc + 1) * 1536 * 16 * 4) + al(8 * nc * 1536 * 4)
    assert binding.bdscan_boundary_states_workspace_size(d, 1) == binding.bdscan_forward_workspace_size(d)
    G = 1536 // 128
    ncb = min(128, 2 * nc)  # the backward's own chunking is bounded by twice the forward's
    expect = (al(8 * 128 * 1536 * 16 * 4) + al(8 * ncb * 1536 * 16 * 4) + al(8 * ncb * 1536 * 4)
              + al(6 * 8 * 2048 * G * 16 * 4) + al(3 * 8 * ncb * 1536 * 16 * 4) + al(2 * 8 * ncb * 1536 * 4))
    assert binding.bdscan_backward_workspace_size(d) == expect
    assert binding.bdscan_forward_workspace_size(_dims(length=60)) == 0  # invalid dims -> 0


FAKE = 1 << 20  # an aligned address that is never dereferenced on the error paths


def _structs(ptr=FAKE):
    c = binding.bdscan_clean(ptr, ptr, ptr, ptr)
    n = binding.bdscan_noisy(ptr, ptr, ptr, ptr, ptr, ptr, ptr)
    p = binding.bdscan_params(ptr, ptr, ptr, ptr)
    return c, n, p


def _fwd(d, c=None, n=None, p=None, y=FAKE, ws=FAKE, wsb=1 << 40):
    c0, n0, p0 = _structs()
    return binding.bdscan_forward(d, c or c0, n or n0, p or p0, y, y, y, ws, wsb, None)


@pytest.mark.parametrize("kw,code,msg", [
    (dict(length=60), binding.BDSCAN_ERR_ARG, "not a multiple of block"),
    (dict(block=0), binding.BDSCAN_ERR_ARG, "block must be positive"),
    (dict(batch=-1), binding.BDSCAN_ERR_ARG, "negative"),
    (dict(d_state=10), binding.BDSCAN_ERR_UNSUPPORTED, "a multiple of 4 up to 64"),
    (dict(d_state=68), binding.BDSCAN_ERR_UNSUPPORTED, "a multiple of 4 up to 64"),
    (dict(d_inner=12), binding.BDSCAN_ERR_UNSUPPORTED, "multiple of 8"),
    (dict(dtype=binding.BDSCAN_F32, out_dtype=binding.BDSCAN_BF16), binding.BDSCAN_ERR_UNSUPPORTED, "f32 inputs"),
    (dict(dtype=7), binding.BDSCAN_ERR_ARG, "bad dtype"),
    (dict(block=512, length=1024), binding.BDSCAN_ERR_UNSUPPORTED, "above 256"),
])
def test_forward_rejects_bad_dims(kw, code, msg):
    assert _fwd(_dims(**kw)) == code
    assert msg in binding.bdscan_last_error()


def test_forward_rejects_bad_pointers_and_small_workspace():
    d = _dims()
    c, n, p = _structs()
    c.dt = None
    assert _fwd(d, c=c) == binding.BDSCAN_ERR_ARG and "clean.dt is NULL" in binding.bdscan_last_error()
    c, n, p = _structs()
    n.C_r = FAKE + 8
    assert _fwd(d, n=n) == binding.BDSCAN_ERR_ARG and "noisy.C_r is not 16-byte aligned" in binding.bdscan_last_error()
    assert _fwd(d, y=FAKE + 4) == binding.BDSCAN_ERR_ARG
    assert _fwd(d, wsb=16) == binding.BDSCAN_ERR_ARG and "workspace" in binding.bdscan_last_error()
    assert binding.bdscan_forward(None, *_structs(), FAKE, FAKE, FAKE, FAKE, 1 << 40, None) == binding.BDSCAN_ERR_ARG


def test_zero_batch_is_a_noop_without_pointers():
    d = _dims(batch=0)
    c, n, p = _structs(None)
    assert binding.bdscan_forward(d, c, n, p, None, None, None, None, 0, None) == binding.BDSCAN_OK


def test_backward_block_limits():
    d = _dims(block=24, length=48)
    c, n, p = _structs()
    gc = binding.bdscan_clean_grads(FAKE, FAKE, FAKE, FAKE)
    gn = binding.bdscan_noisy_grads(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE)
    gp = binding.bdscan_param_grads(FAKE, FAKE, FAKE, FAKE)
    rc = binding.bdscan_backward(d, c, n, p, FAKE, FAKE, FAKE, None, gc, gn, gp, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_UNSUPPORTED and "multiple of 16" in binding.bdscan_last_error()
    rc = binding.bdscan_backward(_dims(block=512, length=1024), c, n, p, FAKE, FAKE, FAKE, None, gc, gn, gp, FAKE,
                                 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_UNSUPPORTED and "backward block 512 above 256" in binding.bdscan_last_error()
    # blocks above 128 tokens keep their segment checkpoints in the workspace
    assert binding.bdscan_backward_workspace_size(_dims(block=256, length=512)) > \
        binding.bdscan_backward_workspace_size(_dims(block=128, length=512))
    gn.dB_r = None
    rc = binding.bdscan_backward(_dims(), c, n, p, FAKE, FAKE, FAKE, None, gc, gn, gp, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "gnoisy.dB_r is NULL" in binding.bdscan_last_error()


def test_active_block_needs_one_block():
    d = _dims(length=32, block=16)
    _, n, p = _structs()
    rc = binding.bdscan_active_block(d, FAKE, n, p, FAKE, None)
    assert rc == binding.BDSCAN_ERR_ARG and "must equal block" in binding.bdscan_last_error()


def test_active_block_adaln_checks():
    d = _dims(length=16, block=16)
    _, n, p = _structs()
    nbytes = binding.bdscan_active_block_adaln_workspace_size(d)
    assert nbytes >= d.batch * 16 * 8 and nbytes % 256 == 0
    mod = binding.bdscan_adaln(FAKE, FAKE, FAKE, 1e-5)
    rc = binding.bdscan_active_block_adaln(_dims(length=32, block=16), FAKE, n, p, mod, FAKE, FAKE, 1 << 20, None)
    assert rc == binding.BDSCAN_ERR_ARG and "must equal block" in binding.bdscan_last_error()
    rc = binding.bdscan_active_block_adaln(d, FAKE, n, p, None, FAKE, FAKE, 1 << 20, None)
    assert rc == binding.BDSCAN_ERR_ARG and "mod is NULL" in binding.bdscan_last_error()
    bad = binding.bdscan_adaln(FAKE, None, FAKE, 1e-5)
    rc = binding.bdscan_active_block_adaln(d, FAKE, n, p, bad, FAKE, FAKE, 1 << 20, None)
    assert rc == binding.BDSCAN_ERR_ARG and "mod.scale is NULL" in binding.bdscan_last_error()
    neg = binding.bdscan_adaln(FAKE, FAKE, FAKE, -1.0)
    rc = binding.bdscan_active_block_adaln(d, FAKE, n, p, neg, FAKE, FAKE, 1 << 20, None)
    assert rc == binding.BDSCAN_ERR_ARG and "eps" in binding.bdscan_last_error()
    rc = binding.bdscan_active_block_adaln(d, FAKE, n, p, mod, FAKE, FAKE, nbytes - 1, None)
    assert rc == binding.BDSCAN_ERR_ARG and "workspace" in binding.bdscan_last_error()


def test_mixer_checks_and_workspace():
    d = _dims()
    c, n, p = _structs()
    mp = binding.bdscan_mixer_params(FAKE, FAKE, FAKE, FAKE)
    fw = binding.bdscan_mixer_forward_workspace_size(d)
    bw = binding.bdscan_mixer_backward_workspace_size(d)
    assert fw > 0 and bw > fw and fw % 256 == 0
    assert binding.bdscan_mixer_boundary_states_workspace_size(d) == fw
    rc = binding.bdscan_mixer_forward(d, c, FAKE, n, FAKE, p, None, FAKE, FAKE, FAKE, FAKE, fw, None)
    assert rc == binding.BDSCAN_ERR_ARG and "mparams is NULL" in binding.bdscan_last_error()
    bad = binding.bdscan_mixer_params(FAKE, None, FAKE, FAKE)
    rc = binding.bdscan_mixer_forward(d, c, FAKE, n, FAKE, p, bad, FAKE, FAKE, FAKE, FAKE, fw, None)
    assert rc == binding.BDSCAN_ERR_ARG and "conv_b" in binding.bdscan_last_error()
    rc = binding.bdscan_mixer_forward(d, c, FAKE, n, FAKE, p, mp, FAKE, FAKE, FAKE, FAKE, fw - 1, None)
    assert rc == binding.BDSCAN_ERR_ARG and "workspace" in binding.bdscan_last_error()
    rc = binding.bdscan_mixer_forward(d, c, None, n, FAKE, p, mp, FAKE, FAKE, FAKE, FAKE, fw, None)
    assert rc == binding.BDSCAN_ERR_ARG and "z_c" in binding.bdscan_last_error()
    # the cache build takes the gate and the clean output together or not at all
    rc = binding.bdscan_mixer_boundary_states(d, c, FAKE, FAKE, FAKE, mp, None, None, None, FAKE, FAKE, 1, FAKE, fw,
                                              None)
    assert rc == binding.BDSCAN_ERR_ARG and "both z_c and out_c" in binding.bdscan_last_error()
    # the active block needs its convolution state
    da = _dims(length=16, block=16)
    rc = binding.bdscan_mixer_active_block(da, FAKE, None, n, FAKE, p, mp, FAKE, FAKE, 1 << 30, None)
    assert rc == binding.BDSCAN_ERR_ARG and "conv_seed" in binding.bdscan_last_error()
    # backward block limits as for bdscan_backward
    db = _dims(length=96, block=24)
    gc = binding.bdscan_clean_grads(FAKE, FAKE, FAKE, FAKE)
    gn = binding.bdscan_noisy_grads(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE)
    gp = binding.bdscan_param_grads(FAKE, FAKE, FAKE, FAKE)
    gm = binding.bdscan_mixer_grads(FAKE, FAKE, FAKE, FAKE)
    rc = binding.bdscan_mixer_backward(db, c, FAKE, n, FAKE, p, mp, FAKE, FAKE, None, gc, FAKE, gn, FAKE, gp, gm, FAKE,
                                       1 << 40, None)
    assert rc == binding.BDSCAN_ERR_UNSUPPORTED and "multiple of 16" in binding.bdscan_last_error()


def test_boundary_states_checks():
    d = _dims()
    c, _, _ = _structs()
    rc = binding.bdscan_boundary_states(d, c, FAKE, FAKE, FAKE + 4, None, FAKE, 1, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "init_state" in binding.bdscan_last_error()
    rc = binding.bdscan_boundary_states(d, c, None, FAKE, None, None, FAKE, 1, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "A_f is NULL" in binding.bdscan_last_error()


def test_full_bidir_checks_and_workspace():
    d = _dims(batch=2, length=64, block=16, d_inner=32, d_state=16)
    al = lambda x: (x + 255) // 256 * 256
    # the chunk states of one direction at a time, and each direction's fp32 output
    assert binding.bdscan_full_bidir_workspace_size(d) == (binding.bdscan_forward_workspace_size(d)
                                                           + 2 * al(2 * 64 * 32 * 4))
    _, n, p = _structs()
    n.dt_r = None
    rc = binding.bdscan_full_bidir_forward(d, n, p, FAKE, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "noisy.dt_r is NULL" in binding.bdscan_last_error()
    _, n, p = _structs()
    rc = binding.bdscan_full_bidir_forward(d, n, p, FAKE, FAKE, 64, None)
    assert rc == binding.BDSCAN_ERR_ARG and "workspace" in binding.bdscan_last_error()
    rc = binding.bdscan_full_bidir_forward(_dims(length=60), n, p, FAKE, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG


def test_fails_loudly_without_a_gpu():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    d = _dims()
    rc = _fwd(d)
    assert rc == binding.BDSCAN_ERR_CUDA
    assert "bdscan_forward" in binding.bdscan_last_error()


def _ssd_dims(**kw):
    base = dict(batch=2, length=512, block=256, heads=4, d_state=128)
    base.update(kw)
    return binding.make_ssd_dims(base["batch"], base["length"], base["block"], base["heads"], base["d_state"],
                                 base.get("head_dim", 64))


def test_ssd_workspace_sizes():
    al = lambda x: (x + 255) // 256 * 256
    d = _ssd_dims(batch=8, length=8192, block=256, heads=26, d_state=128)
    nb = 8192 // 256
    assert binding.bdscan_ssd_forward_workspace_size(d) == al(8 * nb * 26 * 4)
    assert binding.bdscan_ssd_boundary_states_workspace_size(d, 1) == al(8 * nb * 26 * 4)
    assert binding.bdscan_ssd_boundary_states_workspace_size(d, 0) == al(8 * nb * 26 * 4) + al(8 * nb * 26 * 64 * 128 * 4)


@pytest.mark.parametrize("kw,code,msg", [
    (dict(length=500), binding.BDSCAN_ERR_ARG, "not a multiple of block"),
    (dict(block=64, length=512), binding.BDSCAN_ERR_UNSUPPORTED, "128 or 256"),
    (dict(head_dim=32), binding.BDSCAN_ERR_UNSUPPORTED, "head_dim"),
    (dict(d_state=16), binding.BDSCAN_ERR_UNSUPPORTED, "d_state"),
    (dict(batch=-1), binding.BDSCAN_ERR_ARG, "negative"),
])
def test_ssd_rejects_bad_dims(kw, code, msg):
    c, n, p = _structs()
    rc = binding.bdscan_ssd_forward(_ssd_dims(**kw), c, n, p, FAKE, FAKE, FAKE, FAKE, 1 << 40, None)
    assert rc == code and msg in binding.bdscan_last_error()
    assert binding.bdscan_ssd_forward_workspace_size(_ssd_dims(**kw)) == 0


def test_ssd_rejects_bad_pointers():
    d = _ssd_dims()
    c, n, p = _structs()
    n.B_r = None
    rc = binding.bdscan_ssd_forward(d, c, n, p, FAKE, FAKE, FAKE, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "noisy.B_r is NULL" in binding.bdscan_last_error()
    c, n, p = _structs()
    rc = binding.bdscan_ssd_forward(d, c, n, p, FAKE, FAKE, FAKE + 8, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "states is not 16-byte aligned" in binding.bdscan_last_error()
    rc = binding.bdscan_ssd_forward(d, c, n, p, FAKE, FAKE, FAKE, FAKE, 16, None)
    assert rc == binding.BDSCAN_ERR_ARG and "workspace too small" in binding.bdscan_last_error()
    rc = binding.bdscan_ssd_boundary_states(d, c, FAKE, FAKE, FAKE + 4, None, FAKE, 1, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "init_state" in binding.bdscan_last_error()
    rc = binding.bdscan_ssd_active_block(d, FAKE, n, p, FAKE, None)
    assert rc == binding.BDSCAN_ERR_ARG and "must equal block" in binding.bdscan_last_error()
    # an empty batch needs no pointers
    c0, n0, p0 = _structs(None)
    assert binding.bdscan_ssd_forward(_ssd_dims(batch=0), c0, n0, p0, None, None, None, None, 0, None) == 0


def test_ssd_wait_selftest_checks_polls():
    assert binding.bdscan_ssd_wait_selftest(0) == binding.BDSCAN_ERR_ARG
    assert "polls" in binding.bdscan_last_error()


def test_ssd_full_bidir_checks_and_workspace():
    al = lambda x: (x + 255) // 256 * 256
    d = _ssd_dims(batch=2, length=512, block=256, heads=4, d_state=128)
    nb = 2
    assert binding.bdscan_ssd_full_bidir_workspace_size(d) == (al(2 * nb * 4 * 4) + al(2 * nb * 4 * 64 * 128 * 4)
                                                              + al(2 * 512 * 4 * 64 * 4))
    _, n, p = _structs()
    rc = binding.bdscan_ssd_full_bidir_forward(d, n, p, FAKE, FAKE, 64, None)
    assert rc == binding.BDSCAN_ERR_ARG and "workspace too small" in binding.bdscan_last_error()
    n.C_f = None
    rc = binding.bdscan_ssd_full_bidir_forward(d, n, p, FAKE, FAKE, 1 << 40, None)
    assert rc == binding.BDSCAN_ERR_ARG and "noisy.C_f is NULL" in binding.bdscan_last_error()


def _prototypes():
    """name -> number of parameters, from the prototypes of include/*.h."""
    out = {}
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        for m in re.finditer(r"\b(bdscan_\w+)\s*\(([^;{]*?)\)\s*;", text, flags=re.S):
            params = m.group(2).strip()
            out[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_binding_argument_counts_match_the_headers():
    protos = _prototypes()
    assert set(protos) == set(header_functions())
    for name, _, args in binding.SIGNATURES:
        assert len(args) == protos[name], (name, len(args), protos[name])


def test_release_build_has_no_device_checks():
    assert binding.bdscan_debug_build() == 0
    rc = binding.bdscan_debug_set_slack(1)
    assert rc == binding.BDSCAN_ERR_UNSUPPORTED and "release build" in binding.bdscan_last_error()


def test_debug_build_exports_the_same_functions():
    """The debug build (BDSCAN_DEBUG=1) builds, loads, exports every declared
    function, says it is the debug build, and validates on the host exactly
    like the release build (no GPU is touched before a launch)."""
    lib = binding.load(debug=True)
    for name in header_functions():
        assert hasattr(lib, name), name
    assert lib.bdscan_debug_build() == 1
    assert lib.bdscan_debug_set_slack(-1) == binding.BDSCAN_ERR_ARG
    assert b"negative slack" in lib.bdscan_last_error()
    d = binding.make_dims(1, 64, 16, 32, 3, binding.BDSCAN_F32)
    rc = lib.bdscan_forward(ctypes.byref(d), None, None, None, None, None, None, None, 0, None)
    assert rc == binding.BDSCAN_ERR_UNSUPPORTED and b"d_state 3" in lib.bdscan_last_error()


def test_state_groups_size_their_workspaces_and_other_entry_points_refuse_them():
    """d_state 32 runs in state groups for the forward, backward, cache build
    and active block (their workspaces grow with the per-group buffers); the
    other entry points keep d_state 8 or 16."""
    d16, d32 = _dims(d_state=16), _dims(d_state=32)
    assert binding.bdscan_forward_workspace_size(d32) > binding.bdscan_forward_workspace_size(d16) > 0
    assert binding.bdscan_backward_workspace_size(d32) > binding.bdscan_backward_workspace_size(d16) > 0
    assert binding.bdscan_boundary_states_workspace_size(d32, 1) > 0
    assert binding.bdscan_full_bidir_workspace_size(d32) == 0
    assert "not supported here (8 or 16)" in binding.bdscan_last_error()
    assert binding.bdscan_active_block_adaln_workspace_size(d32) == 0
    assert binding.bdscan_mixer_forward_workspace_size(d32) == 0
