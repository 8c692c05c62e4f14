"""The allocation-free QKV projection + RoPE entry point.

Some callers of this library cannot allocate device memory (a plugin in a
serving process whose pool owns every allocation, or a batching worker that
must not call cudaMalloc between requests).  jnx_op_gemm_rope_noalloc keeps
its scratch in a fixed device array inside the library; this file checks,
through the C ABI, that two calls in a row reproduce bit for bit what the
ordinary workspace entry point (jnx_op_gemm with JNX_EPI_ROPE) computes (the
same kernel on the same table), up to the exact size limit of the fixed
array; that requests beyond it and malformed outputs are refused before any
launch; and that a position outside the table is reported through
jnx_op_gemm_rope_noalloc_status with its row left unrotated.  It is named so
that pytest collects it last."""
import numpy as np
import pytest
import torch

from paper_2607_16074_gb300 import jnx as J

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def _stream():
    return torch.cuda.current_stream().cuda_stream


def _rand(shape, seed, std):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(*shape, generator=g) * std).to(torch.bfloat16).cuda()


def _with_workspace(A, W, out, pos, max_pos, rope_cols, hd, epi=J.JNX_EPI_ROPE):
    L = J.lib()
    ws = torch.zeros(L.jnx_op_gemm_workspace_bytes(max_pos, hd), dtype=torch.uint8, device="cuda")
    J.check(L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), A.shape[0], W.shape[0], A.shape[1],
                          epi, out.data_ptr(), out.shape[1], pos.data_ptr(), max_pos,
                          rope_cols, hd, 10000.0, 0, ws.data_ptr(), ws.numel(), _stream()))
    return ws


def _noalloc(A, W, out, pos, max_pos, rope_cols, hd, ldo=None):
    return J.lib().jnx_op_gemm_rope_noalloc(
        A.data_ptr(), W.data_ptr(), A.shape[0], W.shape[0], A.shape[1], out.data_ptr(),
        out.shape[1] if ldo is None else ldo, pos.data_ptr(), max_pos, rope_cols, hd, 10000.0,
        _stream())


# (H, Hkv, hd, rows, max_pos); the last case fills the fixed array exactly:
# max_pos * hd / 2 == JNX_NOALLOC_MAX_ROPE_ENTRIES, with positions near the top
@pytest.mark.parametrize("H,Hkv,hd,M_,max_pos,top", [
    (2, 1, 128, 301, 900, False),
    (4, 2, 64, 77, 320, False),
    (2, 1, 128, 300, J.JNX_NOALLOC_MAX_ROPE_ENTRIES // 64, True),
])
def test_noalloc_matches_workspace_entry_point_twice(H, Hkv, hd, M_, max_pos, top):
    d = 256
    n = (H + 2 * Hkv) * hd
    A = _rand((M_, d), 1, 1.0)
    W = _rand((n, d), 2, 0.05)
    rng = np.random.default_rng(3)
    p = rng.integers(max_pos - 64 if top else 0, max_pos, M_)
    if top:
        p[:8] = max_pos - 1
    pos = torch.tensor(p, dtype=torch.int32).cuda()
    ref = torch.zeros((M_, n), dtype=torch.bfloat16, device="cuda")
    ws = _with_workspace(A, W, ref, pos, max_pos, (H + Hkv) * hd, hd)
    J.check(J.lib().jnx_check_status(ws.data_ptr(), _stream()))
    for call in range(2):
        out = torch.full((M_, n), float("nan"), dtype=torch.bfloat16, device="cuda")
        J.check(_noalloc(A, W, out, pos, max_pos, (H + Hkv) * hd, hd))
        J.check(J.lib().jnx_op_gemm_rope_noalloc_status(_stream()))
        torch.cuda.synchronize()
        assert torch.equal(out, ref), call


def test_noalloc_refuses_requests_beyond_its_fixed_scratch():
    A = _rand((8, 256), 4, 1.0)
    W = _rand((512, 256), 5, 0.05)
    pos = torch.zeros(8, dtype=torch.int32, device="cuda")
    out = torch.zeros((8, 512), dtype=torch.bfloat16, device="cuda")
    too_many = J.JNX_NOALLOC_MAX_ROPE_ENTRIES // 64 + 1  # positions for head_dim 128
    rc = _noalloc(A, W, out, pos, too_many, 384, 128)
    assert rc == J.JNX_ERR_UNSUPPORTED
    assert "scratch" in J.jnx_last_error()
    torch.cuda.synchronize()
    assert torch.all(out == 0)


def test_noalloc_refuses_malformed_outputs_before_any_launch():
    A = _rand((8, 256), 4, 1.0)
    W = _rand((512, 256), 5, 0.05)
    pos = torch.zeros(8, dtype=torch.int32, device="cuda")
    out = torch.zeros((8, 512), dtype=torch.bfloat16, device="cuda")
    # a row stride shorter than the output width, one that is not a
    # multiple of 16 bytes, and rope columns that are not whole heads
    assert _noalloc(A, W, out, pos, 64, 384, 128, ldo=256) == J.JNX_ERR_INVALID_ARG
    assert _noalloc(A, W, out, pos, 64, 384, 128, ldo=516) == J.JNX_ERR_INVALID_ARG
    assert _noalloc(A, W, out, pos, 64, 300, 128) == J.JNX_ERR_INVALID_ARG
    assert _noalloc(A, W, out, pos, 64, 640, 128) == J.JNX_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert torch.all(out == 0)


def test_noalloc_reports_a_position_outside_the_table():
    """Row 5's position is max_pos: the kernel's bounds check records
    JNX_ERR_DEVICE_BOUNDS in the fixed array's status word, skips that row's
    table load and writes it unrotated (the plain projection); every other
    row is the workspace entry point's.  The next read of the status word
    after a good call is JNX_OK again."""
    H, Hkv, hd, M_, max_pos = 2, 1, 128, 64, 128
    n = (H + 2 * Hkv) * hd
    A = _rand((M_, 256), 6, 1.0)
    W = _rand((n, 256), 7, 0.05)
    p = np.arange(M_) % max_pos
    pos_good = torch.tensor(p, dtype=torch.int32).cuda()
    p[5] = max_pos
    pos_bad = torch.tensor(p, dtype=torch.int32).cuda()
    ref = torch.zeros((M_, n), dtype=torch.bfloat16, device="cuda")
    _with_workspace(A, W, ref, pos_good, max_pos, (H + Hkv) * hd, hd)
    plain = torch.zeros((M_, n), dtype=torch.bfloat16, device="cuda")
    _with_workspace(A, W, plain, pos_good, max_pos, (H + Hkv) * hd, hd, epi=J.JNX_EPI_BF16)
    out = torch.full((M_, n), float("nan"), dtype=torch.bfloat16, device="cuda")
    J.check(_noalloc(A, W, out, pos_bad, max_pos, (H + Hkv) * hd, hd))
    rc = J.lib().jnx_op_gemm_rope_noalloc_status(_stream())
    assert rc == J.JNX_ERR_DEVICE_BOUNDS
    rows = [r for r in range(M_) if r != 5]
    assert torch.equal(out[rows], ref[rows])
    assert torch.equal(out[5], plain[5])
    J.check(_noalloc(A, W, out, pos_good, max_pos, (H + Hkv) * hd, hd))
    J.check(J.lib().jnx_op_gemm_rope_noalloc_status(_stream()))
    torch.cuda.synchronize()
    assert torch.equal(out, ref)
