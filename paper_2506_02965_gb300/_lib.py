"""ctypes binding of the C ABI in include/moe.h (argument marshalling only).

Every function here has the name of the C entry point it calls and the same
arguments. Tensors may be passed as torch tensors (their ``data_ptr()`` is used),
as integer device addresses, or as None (NULL). ``stream`` may be a
``torch.cuda.Stream``, an integer handle, or None for the current torch stream.
A non-OK status raises ``MoEError`` carrying moe_last_error().

There is no fallback: if ``libmoe.so`` is missing this module raises on import.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmoe.so")

MOE_OK, MOE_ERR_INVALID_ARG, MOE_ERR_CUDA, MOE_ERR_DEVICE_CHECK, MOE_ERR_TIMEOUT, \
    MOE_ERR_UNSUPPORTED = range(6)
MOE_F32, MOE_BF16 = 0, 1
MOE_PAIRS_OFF, MOE_PAIRS_ALL, MOE_PAIRS_AUTO = 0, 1, 2


class MoEError(RuntimeError):
    def __init__(self, status: int, fn: str, msg: str):
        super().__init__(f"{fn}: status {status} ({msg})")
        self.status = status


class moe_config(ctypes.Structure):
    _fields_ = [
        ("T", ctypes.c_int64),
        ("d_model", ctypes.c_int32),
        ("n_experts", ctypes.c_int32),
        ("d_ff", ctypes.c_int32),
        ("top_k", ctypes.c_int32),
        ("n_parties", ctypes.c_int32),
        ("n_shared", ctypes.c_int32),
        ("d_ff_shared", ctypes.c_int32),
        ("normalize_topk", ctypes.c_int32),
        ("aux_alpha", ctypes.c_float),
        ("dtype", ctypes.c_int32),
    ]


assert ctypes.sizeof(moe_config) == 48


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is missing: build the CUDA library first "
            "(python -m paper_2506_02965_gb300.build); there is no CPU fallback")
    return ctypes.CDLL(LIB_PATH)


_lib = _load()
P = ctypes.c_void_p
_CFG = ctypes.POINTER(moe_config)

# name -> argtypes (after the config pointer where present)
_SIGS = {
    "moe_workspace_size": [_CFG, ctypes.POINTER(ctypes.c_size_t)],
    "moe_route": [_CFG] + [P] * 10,
    "moe_route_from_logits": [_CFG] + [P] * 7,
    "moe_aux_loss": [_CFG] + [P] * 6,
    "moe_dispatch": [_CFG] + [P] * 7 + [ctypes.c_size_t, P],
    "moe_dispatch_noalloc": [_CFG] + [P] * 7,
    "moe_dispatch_owner": [_CFG] + [P] * 10 + [ctypes.c_size_t, P],
    "moe_expert_ffn_fwd": [_CFG] + [P] * 15,
    "moe_combine_fwd": [_CFG] + [P] * 6,
    "moe_combine_bwd": [_CFG] + [P] * 7,
    "moe_expert_ffn_bwd": [_CFG] + [P] * 23,
    "moe_route_bwd": [_CFG] + [P] * 13 + [ctypes.c_size_t, P],
    "moe_dispatch_bwd": [_CFG] + [P] * 6,
    "moe_device_status": [P, ctypes.POINTER(ctypes.c_int32)],
    "moe_set_wait_limit_ns": [ctypes.c_uint64],
    "moe_set_gemm_pairs": [ctypes.c_int],
    "moe_mse_loss": [_CFG] + [P] * 5 + [ctypes.c_size_t, P],
    "moe_expert_ffn_bwd_kernels": [_CFG, ctypes.POINTER(ctypes.c_int32)],
    "moe_sgd_update": [P, P, P, ctypes.c_int64, ctypes.c_int64, P, ctypes.c_float, ctypes.c_int, P],
    "moe_gather_rows": [P, P, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, P, P],
}
for _n, _a in _SIGS.items():
    f = getattr(_lib, _n)
    f.argtypes = _a
    f.restype = ctypes.c_int
for _n in ("moe_status_string",):
    getattr(_lib, _n).argtypes = [ctypes.c_int]
    getattr(_lib, _n).restype = ctypes.c_char_p
for _n in ("moe_last_error", "moe_version"):
    getattr(_lib, _n).argtypes = []
    getattr(_lib, _n).restype = ctypes.c_char_p

EXPORTED = list(_SIGS) + ["moe_status_string", "moe_last_error", "moe_version"]


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(st: int, fn: str):
    if st != MOE_OK:
        raise MoEError(st, fn, _lib.moe_last_error().decode())


def _call(fn: str, cfg, *args, stream=None):
    c = getattr(_lib, fn)
    conv = []
    for a, ty in zip(args, c.argtypes[1:]):
        conv.append(a if ty is ctypes.c_size_t else _ptr(a))
    _check(c(ctypes.byref(cfg), *conv, _stream(stream)), fn)


def make_config(T, d_model, n_experts, d_ff, top_k, n_parties=1, n_shared=0, d_ff_shared=0,
                normalize_topk=0, aux_alpha=0.01, dtype=MOE_BF16) -> moe_config:
    return moe_config(int(T), int(d_model), int(n_experts), int(d_ff), int(top_k), int(n_parties),
                      int(n_shared), int(d_ff_shared), int(normalize_topk), float(aux_alpha),
                      int(dtype))


def moe_version() -> str:
    return _lib.moe_version().decode()


def moe_status_string(s: int) -> str:
    return _lib.moe_status_string(s).decode()


def moe_last_error() -> str:
    return _lib.moe_last_error().decode()


def moe_workspace_size(cfg) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.moe_workspace_size(ctypes.byref(cfg), ctypes.byref(n)), "moe_workspace_size")
    return n.value


def moe_set_wait_limit_ns(ns: int):
    _check(_lib.moe_set_wait_limit_ns(int(ns)), "moe_set_wait_limit_ns")


def moe_set_gemm_pairs(on: int):
    _check(_lib.moe_set_gemm_pairs(int(on)), "moe_set_gemm_pairs")


def moe_device_status(stream=None) -> int:
    code = ctypes.c_int32(0)
    _check(_lib.moe_device_status(_stream(stream), ctypes.byref(code)), "moe_device_status")
    return code.value


def moe_route(cfg, x, w_router, router_bias, party_offsets, logits, probs, topk_idx, topk_w,
              counts, stream=None):
    _call("moe_route", cfg, x, w_router, router_bias, party_offsets, logits, probs, topk_idx,
          topk_w, counts, stream=stream)


def moe_route_from_logits(cfg, logits, party_offsets, probs, topk_idx, topk_w, counts,
                          stream=None):
    _call("moe_route_from_logits", cfg, logits, party_offsets, probs, topk_idx, topk_w, counts,
          stream=stream)


def moe_aux_loss(cfg, probs, counts, party_offsets, loss, aux_coef, stream=None):
    _call("moe_aux_loss", cfg, probs, counts, party_offsets, loss, aux_coef, stream=stream)


def moe_dispatch(cfg, topk_idx, x, offsets, slot_of, token_of, x_perm, workspace,
                 workspace_bytes, stream=None):
    _call("moe_dispatch", cfg, topk_idx, x, offsets, slot_of, token_of, x_perm, workspace,
          int(workspace_bytes), stream=stream)


def moe_dispatch_noalloc(cfg, topk_idx, x, offsets, slot_of, token_of, x_perm, stream=None):
    _call("moe_dispatch_noalloc", cfg, topk_idx, x, offsets, slot_of, token_of, x_perm,
          stream=stream)


def moe_dispatch_owner(cfg, topk_idx, x, party_offsets, group_expert, offsets, slot_of, token_of,
                       x_perm, send_counts, workspace, workspace_bytes, stream=None):
    _call("moe_dispatch_owner", cfg, topk_idx, x, party_offsets, group_expert, offsets, slot_of,
          token_of, x_perm, send_counts, workspace, int(workspace_bytes), stream=stream)


def moe_expert_ffn_fwd(cfg, x_perm, offsets, w1, w2, h_gu, act, y_perm, x=None, ws1=None,
                       ws2=None, h_gu_sh=None, act_sh=None, y_sh=None, group_expert=None,
                       stream=None):
    _call("moe_expert_ffn_fwd", cfg, x_perm, offsets, w1, w2, h_gu, act, y_perm, x, ws1, ws2,
          h_gu_sh, act_sh, y_sh, group_expert, stream=stream)


def moe_expert_ffn_bwd_kernels(cfg) -> int:
    n = ctypes.c_int32(0)
    _check(_lib.moe_expert_ffn_bwd_kernels(ctypes.byref(cfg), ctypes.byref(n)), "moe_expert_ffn_bwd_kernels")
    return int(n.value)


def moe_mse_loss(cfg, out, target, loss, dout, workspace, workspace_bytes, stream=None):
    _call("moe_mse_loss", cfg, out, target, loss, dout, workspace, workspace_bytes, stream=stream)


def moe_sgd_update(w, dw, n_groups, group_elems, group_counts, lr, dtype, w_master=None, stream=None):
    _check(_lib.moe_sgd_update(_ptr(w), _ptr(dw), _ptr(w_master), int(n_groups), int(group_elems),
                               _ptr(group_counts), float(lr), int(dtype), _stream(stream)), "moe_sgd_update")


def moe_gather_rows(src, rows, n_rows, n_src_rows, row_elems, dtype, dst, stream=None):
    _check(_lib.moe_gather_rows(_ptr(src), _ptr(rows), int(n_rows), int(n_src_rows), int(row_elems),
                                int(dtype), _ptr(dst), _stream(stream)), "moe_gather_rows")


def moe_combine_fwd(cfg, y_perm, topk_w, slot_of, y_sh, out, stream=None):
    _call("moe_combine_fwd", cfg, y_perm, topk_w, slot_of, y_sh, out, stream=stream)


def moe_combine_bwd(cfg, dout, y_perm, topk_w, slot_of, dy_perm, dtopk_w, stream=None):
    _call("moe_combine_bwd", cfg, dout, y_perm, topk_w, slot_of, dy_perm, dtopk_w, stream=stream)


def moe_expert_ffn_bwd(cfg, x_perm, offsets, w1, w2, h_gu, act, dy_perm, dh, dx_perm, dw1, dw2,
                       x=None, dout=None, ws1=None, ws2=None, h_gu_sh=None, act_sh=None,
                       dh_sh=None, dx_sh=None, dws1=None, dws2=None, group_expert=None,
                       stream=None):
    _call("moe_expert_ffn_bwd", cfg, x_perm, offsets, w1, w2, h_gu, act, dy_perm, dh, dx_perm,
          dw1, dw2, x, dout, ws1, ws2, h_gu_sh, act_sh, dh_sh, dx_sh, dws1, dws2, group_expert,
          stream=stream)


def moe_route_bwd(cfg, x, w_router, probs, topk_idx, topk_w, dtopk_w, aux_coef, party_offsets,
                  dlogits, dw_router, dbias, dx_router, workspace, workspace_bytes, stream=None):
    _call("moe_route_bwd", cfg, x, w_router, probs, topk_idx, topk_w, dtopk_w, aux_coef,
          party_offsets, dlogits, dw_router, dbias, dx_router, workspace, int(workspace_bytes),
          stream=stream)


def moe_dispatch_bwd(cfg, dx_perm, slot_of, dx_router, dx_sh, dx, stream=None):
    _call("moe_dispatch_bwd", cfg, dx_perm, slot_of, dx_router, dx_sh, dx, stream=stream)
