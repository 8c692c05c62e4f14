"""The allocation-free QKV projection + RoPE entry point.

Some callers of this library cannot allocate device memory (a plugin in a
serving process whose pool owns every allocation, or a batching worker that
must not call cudaMalloc between requests).  jnx_op_gemm_rope_noalloc keeps
its scratch in a fixed device array inside the library; this file checks,
through the C ABI, that two calls in a row reproduce what the ordinary
workspace entry point (jnx_op_gemm with JNX_EPI_ROPE) computes, and that a
request larger than the fixed scratch is refused before any launch.  It is
named so that pytest collects it last."""
import numpy as np
import pytest
import torch

from paper_2607_16074_gb300 import jnx as J
from tests.helpers import rel_err_bf16_out

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def _rand(shape, seed, std):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(*shape, generator=g) * std).to(torch.bfloat16).cuda()


def _with_workspace(A, W, out, pos, max_pos, rope_cols, hd):
    L = J.lib()
    ws = torch.zeros(L.jnx_op_gemm_workspace_bytes(max_pos, hd), dtype=torch.uint8, device="cuda")
    J.check(L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), A.shape[0], W.shape[0], A.shape[1],
                          J.JNX_EPI_ROPE, out.data_ptr(), out.shape[1], pos.data_ptr(), max_pos,
                          rope_cols, hd, 10000.0, 0, ws.data_ptr(), ws.numel(),
                          torch.cuda.current_stream().cuda_stream))


def _noalloc(A, W, out, pos, max_pos, rope_cols, hd):
    return J.lib().jnx_op_gemm_rope_noalloc(
        A.data_ptr(), W.data_ptr(), A.shape[0], W.shape[0], A.shape[1], out.data_ptr(),
        out.shape[1], pos.data_ptr(), max_pos, rope_cols, hd, 10000.0,
        torch.cuda.current_stream().cuda_stream)


@pytest.mark.parametrize("H,Hkv,hd,M_,max_pos", [(2, 1, 128, 301, 900), (4, 2, 64, 77, 320)])
def test_noalloc_matches_workspace_entry_point_twice(H, Hkv, hd, M_, max_pos):
    d = 256
    n = (H + 2 * Hkv) * hd
    A = _rand((M_, d), 1, 1.0)
    W = _rand((n, d), 2, 0.05)
    pos = torch.tensor(np.random.default_rng(3).integers(0, max_pos, M_), dtype=torch.int32).cuda()
    ref = torch.zeros((M_, n), dtype=torch.bfloat16, device="cuda")
    _with_workspace(A, W, ref, pos, max_pos, (H + Hkv) * hd, hd)
    for call in range(2):
        out = torch.full((M_, n), float("nan"), dtype=torch.bfloat16, device="cuda")
        J.check(_noalloc(A, W, out, pos, max_pos, (H + Hkv) * hd, hd))
        torch.cuda.synchronize()
        got = out.float().cpu().numpy()
        want = ref.float().cpu().numpy()
        assert np.isfinite(got).all(), call
        assert rel_err_bf16_out(got, want) < 1e-4, call


def test_noalloc_refuses_requests_beyond_its_fixed_scratch():
    A = _rand((8, 256), 4, 1.0)
    W = _rand((512, 256), 5, 0.05)
    pos = torch.zeros(8, dtype=torch.int32, device="cuda")
    out = torch.zeros((8, 512), dtype=torch.bfloat16, device="cuda")
    too_many = J.JNX_NOALLOC_MAX_ROPE_ENTRIES // 64 + 1  # positions for head_dim 128
    rc = _noalloc(A, W, out, pos, too_many, 384, 128)
    assert rc == J.JNX_ERR_UNSUPPORTED
    assert "scratch" in J.jnx_last_error()
    assert torch.all(out == 0)
