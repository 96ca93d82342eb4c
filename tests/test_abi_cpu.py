"""Host-side checks of the C ABI library (no GPU needed).

The library must load, export every entry point include/moe.h declares, agree with
the binding on the config struct layout, and reject bad arguments on the host
before any CUDA call. The product path must not import the oracle.
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "moe.h")


@pytest.fixture(scope="module")
def L():
    from paper_2506_02965_gb300 import build as b
    if not os.path.exists(b.LIB) or b._stale(b.LIB, os.path.join(b.CSRC, "moe_abi.cu")):
        b.build()
    from paper_2506_02965_gb300 import _lib
    return _lib


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(moe_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(L):
    syms = declared_symbols()
    assert len(syms) >= 16
    for s in syms:
        assert hasattr(L._lib, s), s
        assert s in L.EXPORTED, s


def test_config_struct_layout(L):
    c = L.moe_config
    assert ctypes.sizeof(c) == 48
    names = [f[0] for f in c._fields_]
    hdr = open(HEADER).read()
    body = hdr[hdr.index("typedef struct {\n    int64_t T;"):hdr.index("} moe_config;")]
    order = re.findall(r"\b(T|d_model|n_experts|d_ff|top_k|n_parties|n_shared|d_ff_shared|"
                       r"normalize_topk|aux_alpha|dtype)\b", body)
    assert order == names


def test_status_strings_and_version(L):
    assert L.moe_status_string(0) == "MOE_OK"
    assert L.moe_status_string(4) == "MOE_ERR_TIMEOUT"
    assert "sm_103a" in L.moe_version()


def test_pair_mode_checked_on_host(L):
    for mode in (0, 1, 2):
        L.moe_set_gemm_pairs(mode)
    with pytest.raises(L.MoEError, match="pair mode"):
        L.moe_set_gemm_pairs(3)
    L.moe_set_gemm_pairs(2)  # the default


def test_workspace_size_is_host_only(L):
    cfg = L.make_config(4096, 1024, 16, 2816, 2)
    n = L.moe_workspace_size(cfg)
    assert n >= 4096 // 128 * 16 * 4


@pytest.mark.parametrize("field,value,frag", [
    ("n_experts", 0, "n_experts"), ("top_k", 0, "top_k"),
    ("top_k", 9, "top_k"), ("d_model", 100, "multiples of 128"), ("dtype", 7, "dtype"),
    ("n_parties", 0, "n_parties"), ("normalize_topk", 2, "normalize_topk"), ("T", -1, "T="),
])
def test_bad_config_rejected_on_host(L, field, value, frag):
    cfg = L.make_config(256, 256, 8, 256, 2)
    setattr(cfg, field, value)
    with pytest.raises(L.MoEError) as ei:
        L.moe_route(cfg, 16, 16, None, None, 16, 16, 16, 16, 16, stream=0)
    assert ei.value.status == L.MOE_ERR_INVALID_ARG
    assert frag in L.moe_last_error()


def test_expert_pool_beyond_256_is_unsupported(L):
    """E up to 256 is built; a larger pool is a documented refusal on the host."""
    cfg = L.make_config(256, 256, 257, 256, 2)
    with pytest.raises(L.MoEError) as ei:
        L.moe_route(cfg, 16, 16, None, None, 16, 16, 16, 16, 16, stream=0)
    assert ei.value.status == L.MOE_ERR_UNSUPPORTED
    assert "n_experts=257" in L.moe_last_error()
    assert L.moe_workspace_size(L.make_config(4096, 1024, 256, 512, 8)) > 0


def test_null_and_misaligned_pointers_rejected_on_host(L):
    cfg = L.make_config(256, 256, 8, 256, 2)
    with pytest.raises(L.MoEError) as ei:
        L.moe_route(cfg, None, 16, None, None, 16, 16, 16, 16, 16, stream=0)
    assert ei.value.status == L.MOE_ERR_INVALID_ARG and "x is NULL" in L.moe_last_error()
    with pytest.raises(L.MoEError):
        L.moe_route(cfg, 18, 16, None, None, 16, 16, 16, 16, 16, stream=0)
    assert "16-byte aligned" in L.moe_last_error()
    cfg2 = L.make_config(256, 256, 8, 256, 2, n_parties=2)
    with pytest.raises(L.MoEError):
        L.moe_route(cfg2, 16, 16, None, None, 16, 16, 16, 16, 16, stream=0)
    assert "party_offsets" in L.moe_last_error()
    with pytest.raises(L.MoEError):
        L.moe_dispatch(cfg, 16, 16, 16, 16, 16, 16, 16, 8, stream=0)
    assert "workspace" in L.moe_last_error()
    with pytest.raises(L.MoEError):
        L.moe_set_wait_limit_ns(0)


def test_gather_rows_checks_arguments_on_host(L):
    """moe_gather_rows rejects negative sizes, unknown dtypes, rows whose length is not a
    multiple of 16 bytes (the kernel moves 16-byte vectors) and NULL or misaligned
    pointers before any device work."""
    cases = [((16, 16, -1, 4, 8, L.MOE_BF16, 16), "negative size"),
             ((16, 16, 4, -1, 8, L.MOE_BF16, 16), "negative size"),
             ((16, 16, 4, 4, 8, 9, 16), "dtype"),
             ((16, 16, 4, 4, 6, L.MOE_BF16, 16), "multiple of 16"),
             ((16, 16, 4, 4, 3, L.MOE_F32, 16), "multiple of 16"),
             ((None, 16, 4, 4, 8, L.MOE_BF16, 16), "src is NULL"),
             ((16, None, 4, 4, 8, L.MOE_BF16, 16), "rows is NULL"),
             ((16, 16, 4, 4, 8, L.MOE_BF16, 24), "16-byte aligned")]
    for args, frag in cases:
        with pytest.raises(L.MoEError) as ei:
            L.moe_gather_rows(*args, stream=0)
        assert ei.value.status == L.MOE_ERR_INVALID_ARG and frag in L.moe_last_error(), frag
    L.moe_gather_rows(None, None, 0, 0, 8, L.MOE_BF16, None, stream=0)  # nothing to move: OK


def test_training_calls_check_arguments_on_host(L):
    """moe_sgd_update and moe_mse_loss reject bad arguments before any device work."""
    cases = [((16, 16, -1, 8, None, 0.1, L.MOE_BF16), "negative size"),
             ((16, 16, 70000, 8, None, 0.1, L.MOE_BF16), "65535"),
             ((16, 16, 2, 8, None, float("nan"), L.MOE_F32), "lr"),
             ((16, 16, 2, 8, None, float("inf"), L.MOE_F32), "lr"),
             ((16, 16, 2, 8, None, 0.1, 7), "dtype"),
             ((None, 16, 2, 8, None, 0.1, L.MOE_F32), "w is NULL")]
    for args, frag in cases:
        with pytest.raises(L.MoEError) as ei:
            L.moe_sgd_update(*args, stream=0)
        assert ei.value.status == L.MOE_ERR_INVALID_ARG and frag in L.moe_last_error(), frag
    L.moe_sgd_update(None, None, 0, 8, None, 0.1, L.MOE_F32, stream=0)  # nothing to do: OK
    cfg = L.make_config(256, 256, 8, 256, 2)
    with pytest.raises(L.MoEError):
        L.moe_mse_loss(cfg, 16, 16, 16, 16, 16, 8, stream=0)
    assert "workspace_bytes" in L.moe_last_error()
    with pytest.raises(L.MoEError):
        L.moe_mse_loss(cfg, 16, None, 16, 16, 16, 4096, stream=0)
    assert "target is NULL" in L.moe_last_error()


def test_backward_kernel_count_follows_the_tile_mode(L):
    """moe_expert_ffn_bwd_kernels (host only): in the default mode the dA GEMM shares a
    launch with dW2 and dX runs as CTA pairs beside a separate dW1 launch (3); with
    single-CTA tiles both pairs of GEMMs share launches (2); fp32 runs four; with
    d = 2048 and F = 1408 every backward GEMM of the routed and the shared experts runs as
    its own pair launch (dA and dX as pairs with a ragged last N-tile, 8); nothing to do,
    no GEMM."""
    mid = L.make_config(4096, 1024, 16, 2816, 2)
    assert L.moe_expert_ffn_bwd_kernels(mid) == 3
    try:
        L.moe_set_gemm_pairs(L.MOE_PAIRS_OFF)
        assert L.moe_expert_ffn_bwd_kernels(mid) == 2
        L.moe_set_gemm_pairs(L.MOE_PAIRS_ALL)
        assert L.moe_expert_ffn_bwd_kernels(mid) == 4
    finally:
        L.moe_set_gemm_pairs(L.MOE_PAIRS_AUTO)
    assert L.moe_expert_ffn_bwd_kernels(L.make_config(512, 256, 8, 512, 2, dtype=L.MOE_F32)) == 4
    assert L.moe_expert_ffn_bwd_kernels(L.make_config(8192, 2048, 64, 1408, 6, n_shared=2,
                                                      d_ff_shared=1408)) == 8
    assert L.moe_expert_ffn_bwd_kernels(L.make_config(0, 1024, 16, 2816, 2)) == 0


def test_binding_refuses_to_load_without_library(L, monkeypatch):
    monkeypatch.setattr(L, "LIB_PATH", "/nonexistent/libmoe.so")
    with pytest.raises(ImportError):
        L._load()


def test_product_path_does_not_touch_the_oracle():
    pkg = os.path.join(ROOT, "paper_2506_02965_gb300")
    for dp, _, fs in os.walk(pkg):
        for f in fs:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dp, f)).read()
                assert not re.search(r"^\s*(from|import)\s+oracle", src, re.M), f
                assert "oracle/" not in src, f
