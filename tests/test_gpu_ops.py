"""Stage-wise parity of each CUDA kernel against the fp64 oracle, through the
C ABI (jnx_ops.h).  Sizes span several tiles and a ragged tail."""
import ctypes as C
import math

import numpy as np
import pytest
import torch

import synth
from oracle import model as M
from oracle import plan as OP
from paper_2607_16074_gb300 import jnx as J
from paper_2607_16074_gb300 import runtime as R
from tests.gpu_helpers import bits, f64, randn_bf16, stream
from tests import bf16_emulation as E
from tests.helpers import BF16_TOL, check_bf16_out, oracle_requests, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def _gemm(A, W, epi, out, ldo, pos=None, max_pos=0, rope_cols=0, hd=0, act=0, ws=None):
    L = J.lib()
    J.check(L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), A.shape[0], W.shape[0], A.shape[1], epi,
                          out.data_ptr(), ldo, pos.data_ptr() if pos is not None else None,
                          max_pos, rope_cols, hd, 10000.0, act,
                          ws.data_ptr() if ws is not None else None,
                          ws.numel() if ws is not None else 0, stream()))


@pytest.mark.parametrize("M_,N_,K_", [(1, 256, 64), (127, 256, 128), (300, 768, 256),
                                       (1000, 512, 1024), (257, 1536, 4096)])
def test_gemm_f32_and_bf16(M_, N_, K_):
    A = randn_bf16((M_, K_), 1)
    W = randn_bf16((N_, K_), 2, 0.05)
    ref = f64(A) @ f64(W).T
    out = torch.full((M_, N_), float("nan"), device="cuda")
    _gemm(A, W, J.JNX_EPI_F32, out, N_)
    torch.cuda.synchronize()
    # fp32 accumulation of exact bf16 products
    e32 = rel_err(f64(out), ref)
    assert e32 < 1e-4, e32   # fp32 accumulation over K terms
    ob = torch.zeros((M_, N_), dtype=torch.bfloat16, device="cuda")
    _gemm(A, W, J.JNX_EPI_BF16, ob, N_)
    check_bf16_out(f64(ob), ref, 1e-4, f"gemm bf16 {M_}x{N_}x{K_}")


def test_gemm_residual_epilogue():
    M_, N_, K_ = 333, 512, 320
    A, W = randn_bf16((M_, K_), 3), randn_bf16((N_, K_), 4, 0.05)
    x0 = torch.randn((M_, N_), generator=torch.Generator().manual_seed(5)).cuda()
    x = x0.clone()
    _gemm(A, W, J.JNX_EPI_RESID, x, N_)
    ref = f64(x0) + f64(A) @ f64(W).T
    assert rel_err(f64(x), ref) < 1e-5


@pytest.mark.parametrize("glu", [J.JNX_GLU_SWIGLU, J.JNX_GLU_GEGLU_TANH])
def test_gemm_glu_epilogue(glu):
    M_, F, K_ = 200, 384, 256
    A = randn_bf16((M_, K_), 6)
    Wg, Wu = randn_bf16((F, K_), 7, 0.1), randn_bf16((F, K_), 8, 0.1)
    Wgu = torch.empty((2 * F, K_), dtype=torch.bfloat16, device="cuda")
    J.check(J.lib().jnx_pack_gate_up(Wg.data_ptr(), Wu.data_ptr(), F, K_, Wgu.data_ptr(),
                                     stream()))
    out = torch.zeros((M_, F), dtype=torch.bfloat16, device="cuda")
    _gemm(A, Wgu, J.JNX_EPI_GLU, out, F, act=glu)
    g = f64(A) @ f64(Wg).T
    u = f64(A) @ f64(Wu).T
    ref = (M.silu(g) if glu == 0 else M.gelu_tanh(g)) * u
    check_bf16_out(f64(out), ref, 1e-3, f"gemm glu {glu}")


@pytest.mark.parametrize("H,Hkv,hd", [(4, 4, 64), (2, 2, 128), (2, 1, 256), (4, 2, 128)])
def test_gemm_rope_epilogue(H, Hkv, hd):
    d = 256
    n = (H + 2 * Hkv) * hd
    if n % 256:
        pytest.skip("fused width not a multiple of 256")
    M_ = 301
    A = randn_bf16((M_, d), 9)
    W = randn_bf16((n, d), 10, 0.05)
    pos = torch.tensor(np.random.default_rng(0).integers(0, 900, M_), dtype=torch.int32).cuda()
    ws = torch.zeros(J.lib().jnx_op_gemm_workspace_bytes(900, hd), dtype=torch.uint8,
                     device="cuda")
    out = torch.zeros((M_, n), dtype=torch.bfloat16, device="cuda")
    _gemm(A, W, J.JNX_EPI_ROPE, out, n, pos=pos, max_pos=900, rope_cols=(H + Hkv) * hd, hd=hd,
          ws=ws)
    y = f64(A) @ f64(W).T
    p = pos.cpu().numpy()
    q = M.rope(y[:, :H * hd].reshape(M_, H, hd), p, 1e4).reshape(M_, -1)
    k = M.rope(y[:, H * hd:(H + Hkv) * hd].reshape(M_, Hkv, hd), p, 1e4).reshape(M_, -1)
    ref = np.concatenate([q, k, y[:, (H + Hkv) * hd:]], axis=1)
    check_bf16_out(f64(out), ref, 1e-4, f"gemm rope {H}/{Hkv}/{hd}")


def test_gemm_full_size_sampled_rows():
    """The 7B-class gate/up GEMM at its full launch size (M = 65817 packed
    tokens, N = 2 x 11008, K = 4096), checked on sampled rows."""
    M_, F, K_ = 65817, 11008, 4096
    A = randn_bf16((M_, K_), 11)
    Wg, Wu = randn_bf16((F, K_), 12, 0.02), randn_bf16((F, K_), 13, 0.02)
    Wgu = torch.empty((2 * F, K_), dtype=torch.bfloat16, device="cuda")
    J.check(J.lib().jnx_pack_gate_up(Wg.data_ptr(), Wu.data_ptr(), F, K_, Wgu.data_ptr(),
                                     stream()))
    out = torch.zeros((M_, F), dtype=torch.bfloat16, device="cuda")
    _gemm(A, Wgu, J.JNX_EPI_GLU, out, F, act=0)
    torch.cuda.synchronize()
    rows = np.r_[0, 1, 127, 128, 40000, M_ - 2, M_ - 1, np.random.default_rng(1).integers(0, M_, 9)]
    a = f64(A[rows])
    g, u = a @ f64(Wg).T, a @ f64(Wu).T
    check_bf16_out(f64(out[rows]), M.silu(g) * u, 1e-3, "gate/up glu full size")


def test_rmsnorm():
    for d in (256, 1024, 4096):
        Mr = 77
        x = torch.randn((Mr, d), generator=torch.Generator().manual_seed(d)).cuda() * 3
        gam = randn_bf16((d,), d + 1, 0.02) + 1
        gam = gam.to(torch.bfloat16)
        out = torch.zeros((Mr, d), dtype=torch.bfloat16, device="cuda")
        J.check(J.lib().jnx_op_rmsnorm(x.data_ptr(), gam.data_ptr(), 1e-6, Mr, d, out.data_ptr(),
                                       stream()))
        ref = M.rmsnorm(f64(x), bits(gam), 1e-6)
        check_bf16_out(f64(out), ref, 1e-4, f"rmsnorm d={d}")


def _ragged_cu(lengths):
    return np.concatenate([[0], np.cumsum(lengths)]).astype(np.int32)


@pytest.mark.parametrize("H,Hkv,hd", [(4, 4, 64), (2, 2, 128), (4, 1, 256), (4, 2, 128)])
def test_attention_varlen(H, Hkv, hd):
    # lengths straddle the 64- and 128-key tiles and the 128-query tile
    lengths = [1, 17, 64, 65, 127, 128, 129, 200, 3, 300]
    cu = _ragged_cu(lengths)
    N = int(cu[-1])
    qkv = randn_bf16((N, (H + 2 * Hkv) * hd), 20 + hd, 1.0)
    out = torch.full((N, H * hd), 7.0, dtype=torch.bfloat16, device="cuda")
    cu_d = torch.tensor(cu).cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    J.check(J.lib().jnx_op_attention(qkv.data_ptr(), N, H, Hkv, hd, cu_d.data_ptr(), len(lengths),
                                     max(lengths), out.data_ptr(), st.data_ptr(), stream()))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    X = f64(qkv)
    for s in range(len(lengths)):
        a, b = cu[s], cu[s + 1]
        q = X[a:b, :H * hd].reshape(-1, H, hd)
        k = X[a:b, H * hd:(H + Hkv) * hd].reshape(-1, Hkv, hd)
        v = X[a:b, (H + Hkv) * hd:].reshape(-1, Hkv, hd)
        ref = M.attention(q, k, v).reshape(b - a, -1)
        # floor: P and the output in bf16 (tests/bf16_emulation.py)
        fl = rel_err(E.attention(q, k, v), ref)
        check_bf16_out(f64(out[a:b]), ref, BF16_TOL, f"attention {H}/{Hkv}/{hd} sample {s}", fl)


def test_attention_sharp_logits():
    # large logits: attention nearly one-hot, exercises the online max
    H, Hkv, hd = 2, 2, 128
    lengths = [150, 90]
    cu = _ragged_cu(lengths)
    N = int(cu[-1])
    qkv = randn_bf16((N, (H + 2 * Hkv) * hd), 31, 3.0)
    out = torch.zeros((N, H * hd), dtype=torch.bfloat16, device="cuda")
    J.check(J.lib().jnx_op_attention(qkv.data_ptr(), N, H, Hkv, hd,
                                     torch.tensor(cu).cuda().data_ptr(), 2, 150, out.data_ptr(),
                                     None, stream()))
    torch.cuda.synchronize()
    X = f64(qkv)
    for s in range(2):
        a, b = cu[s], cu[s + 1]
        q, k, v = (X[a:b, :256].reshape(-1, H, hd), X[a:b, 256:512].reshape(-1, H, hd),
                   X[a:b, 512:].reshape(-1, H, hd))
        ref = M.attention(q, k, v).reshape(b - a, -1)
        fl = rel_err(E.attention(q, k, v), ref)
        check_bf16_out(f64(out[a:b]), ref, BF16_TOL, f"attention sharp sample {s}", fl)


def test_final_pool():
    d = 1024
    lengths = [5, 300, 1, 64]
    cu = _ragged_cu(lengths)
    N = int(cu[-1])
    x = torch.randn((N, d), generator=torch.Generator().manual_seed(3)).cuda() * 2
    gam = (randn_bf16((d,), 4, 0.02) + 1).to(torch.bfloat16)
    pooled = torch.zeros((4, d), device="cuda")
    hidden = torch.zeros((N, d), dtype=torch.bfloat16, device="cuda")
    J.check(J.lib().jnx_op_final_pool(x.data_ptr(), gam.data_ptr(), 1e-6,
                                      torch.tensor(cu).cuda().data_ptr(), 4, d, pooled.data_ptr(),
                                      hidden.data_ptr(), stream()))
    torch.cuda.synchronize()
    h = M.rmsnorm(f64(x), bits(gam), 1e-6)
    check_bf16_out(f64(hidden), h, 1e-4, "final norm rows")
    for s in range(4):
        e = rel_err(f64(pooled[s]), M.mean_pool(h[cu[s]:cu[s + 1]]))
        assert e < 1e-4, (s, e)


def test_pack_bit_exact_and_bounds():
    w = synth.make_workload("tiny")
    bw = synth.make_backbone_weights(w)
    inp = synth.make_inputs(w)
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), 2, 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    vis, tid, tab = inp["vision"].cuda(), inp["text_ids"].cuda(), bw["text_table"].cuda()
    x = torch.full((plan.n_tokens, w.backbone.d), float("nan"), device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    J.check(J.lib().jnx_op_pack(g.ref, vis.data_ptr(), vis.shape[0], tid.data_ptr(),
                                tid.shape[0], tab.data_ptr(), w.backbone.vocab, w.backbone.d,
                                x.data_ptr(), st.data_ptr(), stream()))
    torch.cuda.synchronize()
    bb = M.backbone_dict(w)
    npi = synth.to_numpy_tree(inp)
    order = [s for t in plan.slot_tenant.tolist() for r in w.requests if r.tenant == t
             for s in r.samples]
    ref = np.concatenate([M.sample_embeddings(bb, vars(s), npi["vision"], npi["text_ids"],
                                              synth.bf16_bits(bw["text_table"]))
                          for s in order])
    assert np.array_equal(f64(x), ref)
    assert int(st.item()) == 0
    # a vision buffer shorter than the plan needs: zero rows + status
    J.check(J.lib().jnx_op_pack(g.ref, vis.data_ptr(), 100, tid.data_ptr(), tid.shape[0],
                                tab.data_ptr(), w.backbone.vocab, w.backbone.d, x.data_ptr(),
                                st.data_ptr(), stream()))
    torch.cuda.synchronize()
    assert int(st.item()) == J.JNX_ERR_DEVICE_BOUNDS
    src = plan.gather_src
    bad = np.where(src >= 100)[0]
    assert bad.size and torch.all(x[torch.tensor(bad).cuda()] == 0)
    good = np.where((src >= 0) & (src < 100))[0]
    assert np.array_equal(f64(x[torch.tensor(good).cuda()]), ref[good])


def test_pack_bit_exact_at_the_7b_class_width():
    """The packer over the whole 7B-class group (65,817 rows of d = 4096,
    222 samples of 32 tenants) against the oracle's per-sample embeddings in
    packed order, bit for bit."""
    w = synth.make_workload("llama7b")
    inp = synth.make_inputs(w, device="cuda")
    tab = synth._normal((w.backbone.vocab, w.backbone.d), 1.0, "cuda", w.seed, 31)
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    x = torch.full((plan.n_tokens, w.backbone.d), float("nan"), device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    J.check(J.lib().jnx_op_pack(g.ref, inp["vision"].data_ptr(), inp["vision"].shape[0],
                                inp["text_ids"].data_ptr(), inp["text_ids"].shape[0],
                                tab.data_ptr(), w.backbone.vocab, w.backbone.d, x.data_ptr(),
                                st.data_ptr(), stream()))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    bb = M.backbone_dict(w)
    npi = synth.to_numpy_tree(inp)
    table = synth.bf16_bits(tab)
    order = [s for t in plan.slot_tenant.tolist() for r in w.requests if r.tenant == t
             for s in r.samples]
    got = x.cpu().numpy()
    row = 0
    for s in order:
        ref = M.sample_embeddings(bb, vars(s), npi["vision"], npi["text_ids"], table)
        assert np.array_equal(got[row:row + ref.shape[0]], ref.astype(np.float32)), row
        row += ref.shape[0]
    assert row == plan.n_tokens
