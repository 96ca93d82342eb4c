"""Shared fixtures/helpers of the GPU tests (device buffers from numpy)."""
import numpy as np
import pytest


def need_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2506_02965_gb300 import _lib
    return _lib


def dev(a, dtype):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dtype)


def empty(shape, dtype):
    import torch
    return torch.empty(*shape, dtype=dtype, device="cuda")


def tdt(shape):
    import torch
    return torch.bfloat16 if shape.dtype == "bf16" else torch.float32


def cfg_of(L, sh):
    return L.make_config(sh.T, sh.d_model, sh.n_experts, sh.d_ff, sh.top_k, sh.n_parties,
                         sh.n_shared, sh.d_ff_shared, sh.normalize_topk, sh.aux_alpha,
                         L.MOE_BF16 if sh.dtype == "bf16" else L.MOE_F32)


def status(L):
    import torch
    torch.cuda.synchronize()
    return L.moe_device_status(None)
