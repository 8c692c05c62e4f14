"""Helpers for GPU tests: seeded test tensors and conversions for the oracle."""
import numpy as np
import torch

from oracle import model as M


def dev():
    return torch.device("cuda")


def randn_bf16(shape, seed, std=1.0, device="cuda"):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(*shape, generator=g) * std).to(torch.bfloat16).to(device)


def f64(t):
    """A torch tensor (any dtype, any device) as a float64 numpy array (exact
    for bf16/fp32)."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def ptr(t):
    return t.data_ptr()


def stream():
    return torch.cuda.current_stream().cuda_stream
