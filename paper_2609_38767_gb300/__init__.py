"""GB300 (sm_103a) training-data-attribution hot path of the dattri-LLM paper.

Python binding of the C ABI in ``include/tda.h``: every function here has the
name and argument order of its C entry point and only marshals arguments
(torch tensors become device pointers, ``stream=None`` becomes torch's current
CUDA stream). All computation happens in ``libtda.so``. Importing this package
loads nothing; the first call loads the library and raises if it is missing,
so there is no silent CPU path.
"""
from __future__ import annotations

import ctypes
import os
import threading

__all__ = [
    "LayerDesc", "TdaError", "load", "tda_proj_entries", "tda_workspace_size", "tda_project",
    "tda_project_engine", "tda_project_host_ws_min", "tda_project_host", "tda_noalloc_scratch_bytes",
    "tda_project_materialized_noalloc",
    "tda_similarity_projected", "tda_similarity_exact", "tda_norms", "tda_cosine", "tda_kfac_state_bytes", "tda_kfac_workspace_size",
    "tda_kfac_reset", "tda_kfac_accumulate_factors", "tda_project_kfac", "tda_kfac_eigen",
    "tda_kfac_accumulate_eigenvalues", "tda_kfac_apply",
    "tda_token_scores_workspace_size", "tda_token_scores", "tda_mask_gather", "tda_precondition_state_bytes", "tda_precondition",
    "tda_precondition_info", "tda_score", "tda_score_engine", "tda_similarity_gram_engine", "tda_topk", "tda_route", "tda_route_calibrate",
    "tda_route_set_model", "tda_device_status", "tda_selftest_bounded_wait", "tda_last_error", "tda_version", "tda_launch_count",
    "tda_set_sm_budget", "tda_get_sm_budget",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
_lock = threading.Lock()
_lib = None

# enums of include/tda.h
TDA_OK, TDA_ERR_INVALID_ARG, TDA_ERR_UNSUPPORTED, TDA_ERR_WORKSPACE = 0, 1, 2, 3
TDA_ERR_CUDA, TDA_ERR_NOT_SPD, TDA_ERR_TIMEOUT = 4, 5, 6
TDA_F32, TDA_BF16, TDA_F64 = 0, 1, 2
TDA_PROJ_RADEMACHER, TDA_PROJ_IDENTITY = 0, 1
TDA_ROUTE_AUTO, TDA_ROUTE_FACTORED, TDA_ROUTE_MATERIALIZE, TDA_ROUTE_GRAM = -1, 0, 1, 2
TDA_OP_PROJECT, TDA_OP_SIMILARITY_PROJECTED, TDA_OP_SIMILARITY_EXACT = 0, 1, 2
TDA_OP_NORM_PROJECTED, TDA_OP_NORM_EXACT = 3, 4
TDA_PC_RESET, TDA_PC_FIT_ACCUM, TDA_PC_FACTOR, TDA_PC_APPLY, TDA_PC_FACTOR_APPLY = 0, 1, 2, 3, 4
TDA_KFAC, TDA_EKFAC = 0, 1
TDA_CALIBRATE_WS_BYTES = 768 << 20
_STATUS = {0: "TDA_OK", 1: "TDA_ERR_INVALID_ARG", 2: "TDA_ERR_UNSUPPORTED", 3: "TDA_ERR_WORKSPACE",
           4: "TDA_ERR_CUDA", 5: "TDA_ERR_NOT_SPD", 6: "TDA_ERR_TIMEOUT"}


class LayerDesc(ctypes.Structure):
    """tda_layer_desc."""
    _fields_ = [("d_in", ctypes.c_int64), ("d_out", ctypes.c_int64), ("T", ctypes.c_int64),
                ("k_in", ctypes.c_int32), ("k_out", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("layer", ctypes.c_uint32), ("kind", ctypes.c_int32)]

    def __init__(self, d_in, d_out, T, k_in, k_out, seed=0, layer=0, kind=TDA_PROJ_RADEMACHER):
        super().__init__(d_in, d_out, T, k_in, k_out, seed, layer, kind)


class TdaError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


def lib_path(name: str = "libtda.so") -> str:
    return os.path.join(_HERE, name)


def load() -> ctypes.CDLL:
    """Load libtda.so (built by ``build.build()``); raises if it is absent."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = lib_path()
        if not os.path.exists(path):
            raise ImportError(f"{path} is missing: run paper_2609_38767_gb300.build.build() first")
        lib = ctypes.CDLL(path)
        P, I32, I64, U32, U64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32, ctypes.c_uint64
        D, F, SZ = ctypes.c_double, ctypes.c_float, ctypes.c_size_t
        LP = ctypes.POINTER(LayerDesc)
        sig = {
            "tda_proj_entries": (I32, [U64, U32, I32, I32, I64, I32, P, P]),
            "tda_workspace_size": (I32, [I32, LP, I32, I64, I64, I32, ctypes.POINTER(SZ)]),
            "tda_project": (I32, [LP, I32, P, P, I64, P, I64, I32, P, SZ, P]),
            "tda_project_engine": (I32, [LP, I32, P, P]),
            "tda_project_host_ws_min": (SZ, [LP, I32]),
            "tda_project_host": (I32, [LP, I32, P, P, I64, P, I64, P, SZ, P]),
            "tda_noalloc_scratch_bytes": (SZ, []),
            "tda_project_materialized_noalloc": (I32, [LP, I32, P, P, I64, P, I64, P]),
            "tda_similarity_projected": (I32, [LP, I32, P, P, I64, P, P, I64, P, I64, F, I32, P, SZ, P]),
            "tda_norms": (I32, [I32, LP, I32, P, P, I64, P, I32, P, SZ, P]),
            "tda_cosine": (I32, [P, I64, I64, I64, P, P, P]),
            "tda_similarity_exact": (I32, [LP, I32, P, P, I64, P, P, I64, P, I64, F, I32, P, SZ, P]),
            "tda_precondition_state_bytes": (SZ, [I64, I32]),
            "tda_kfac_state_bytes": (SZ, [I32, I32]),
            "tda_token_scores_workspace_size": (SZ, [LP]),
            "tda_token_scores": (I32, [LP, I32, P, P, I64, P, I64, I64, P, I64, F, P, SZ, P]),
            "tda_mask_gather": (I32, [LP, I32, P, P, I64, P, P, I64, P, I64, P]),
            "tda_kfac_workspace_size": (SZ, [LP, I32]),
            "tda_kfac_reset": (I32, [I32, I32, I32, P, P]),
            "tda_kfac_accumulate_factors": (I32, [LP, I32, P, P, I64, P, P, SZ, P]),
            "tda_project_kfac": (I32, [LP, I32, P, P, I64, P, I64, P, P, SZ, P]),
            "tda_kfac_eigen": (I32, [I32, I32, I32, P, P]),
            "tda_kfac_accumulate_eigenvalues": (I32, [I32, I32, I32, P, P, I64, I64, P, SZ, P]),
            "tda_kfac_apply": (I32, [I32, I32, I32, I32, P, D, D, P, I64, I64, P, I64, P]),
            "tda_precondition": (I32, [I32, I32, I64, I32, P, P, I64, I64, I64, D, D, P, I64, I64, P, I64, P]),
            "tda_precondition_info": (I32, [I32, I64, I32, P, ctypes.POINTER(D), P]),
            "tda_score": (I32, [P, I32, I64, I64, P, I64, I64, I64, P, I64, F, P]),
            "tda_topk": (I32, [P, I64, I64, I64, I32, P, P, P]),
            "tda_score_engine": (I32, [P, I32, I64, I64, P, I64, I64, I64]),
            "tda_similarity_gram_engine": (I32, [LP, I32, P, P, P, P]),
            "tda_route": (I32, [LP, I32, I64, I64, I32, ctypes.POINTER(I32), ctypes.POINTER(D)]),
            "tda_route_calibrate": (I32, [P, SZ, P, ctypes.POINTER(D)]),
            "tda_route_set_model": (I32, [I32]),
            "tda_device_status": (I32, [P]),
            "tda_selftest_bounded_wait": (I32, [U64, P]),
            "tda_last_error": (ctypes.c_char_p, []),
            "tda_version": (I32, []),
            "tda_launch_count": (U64, []),
            "tda_set_sm_budget": (I32, [I32]),
            "tda_get_sm_budget": (I32, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _ptr(x):
    """Device (or host) address of a tensor, an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status: int) -> None:
    if status != TDA_OK:
        raise TdaError(status, load().tda_last_error().decode())


def tda_last_error() -> str:
    return load().tda_last_error().decode()


def tda_version() -> int:
    return int(load().tda_version())


def tda_launch_count() -> int:
    return int(load().tda_launch_count())


def tda_set_sm_budget(n_sms: int) -> None:
    _check(load().tda_set_sm_budget(n_sms))


def tda_get_sm_budget() -> int:
    return int(load().tda_get_sm_budget())


def tda_proj_entries(seed, layer, side, kind, rows, cols, out, stream=None):
    _check(load().tda_proj_entries(seed, layer, side, kind, rows, cols, _ptr(out), _stream(stream)))


def tda_workspace_size(op, L, dtype, n1, n2, route=TDA_ROUTE_AUTO) -> int:
    b = ctypes.c_size_t(0)
    _check(load().tda_workspace_size(op, ctypes.byref(L), dtype, n1, n2, route, ctypes.byref(b)))
    return int(b.value)


def tda_project(L, dtype, A, B, N, phi, ld_phi, route=TDA_ROUTE_AUTO, ws=None, ws_bytes=0, stream=None):
    _check(load().tda_project(ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(phi), ld_phi, route,
                              _ptr(ws), ws_bytes, _stream(stream)))


def tda_project_engine(L, dtype, A, B) -> int:
    return int(load().tda_project_engine(ctypes.byref(L), dtype, _ptr(A), _ptr(B)))


def tda_project_host_ws_min(L, dtype) -> int:
    return int(load().tda_project_host_ws_min(ctypes.byref(L), dtype))


def tda_project_host(L, dtype, A_h, B_h, N, phi, ld_phi, ws, ws_bytes, stream=None):
    _check(load().tda_project_host(ctypes.byref(L), dtype, _ptr(A_h), _ptr(B_h), N, _ptr(phi), ld_phi,
                                   _ptr(ws), ws_bytes, _stream(stream)))


def tda_noalloc_scratch_bytes() -> int:
    return int(load().tda_noalloc_scratch_bytes())


def tda_project_materialized_noalloc(L, dtype, A, B, N, phi, ld_phi, stream=None):
    _check(load().tda_project_materialized_noalloc(ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(phi),
                                                   ld_phi, _stream(stream)))


def tda_similarity_projected(L, dtype, Aq, Bq, n_q, At, Bt, n_t, S, ld_S, beta=0.0, route=TDA_ROUTE_AUTO,
                             ws=None, ws_bytes=0, stream=None):
    _check(load().tda_similarity_projected(ctypes.byref(L), dtype, _ptr(Aq), _ptr(Bq), n_q, _ptr(At), _ptr(Bt),
                                           n_t, _ptr(S), ld_S, beta, route, _ptr(ws), ws_bytes, _stream(stream)))


def tda_norms(op, L, dtype, A, B, N, out, route=TDA_ROUTE_AUTO, ws=None, ws_bytes=0, stream=None):
    _check(load().tda_norms(op, ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(out), route, _ptr(ws), ws_bytes,
                            _stream(stream)))


def tda_cosine(S, n_q, n_t, ld_S, nq, nt, stream=None):
    _check(load().tda_cosine(_ptr(S), n_q, n_t, ld_S, _ptr(nq), _ptr(nt), _stream(stream)))


def tda_similarity_exact(L, dtype, Aq, Bq, n_q, At, Bt, n_t, S, ld_S, beta=0.0, route=TDA_ROUTE_AUTO,
                         ws=None, ws_bytes=0, stream=None):
    _check(load().tda_similarity_exact(ctypes.byref(L), dtype, _ptr(Aq), _ptr(Bq), n_q, _ptr(At), _ptr(Bt),
                                       n_t, _ptr(S), ld_S, beta, route, _ptr(ws), ws_bytes, _stream(stream)))


def tda_token_scores_workspace_size(L) -> int:
    return int(load().tda_token_scores_workspace_size(ctypes.byref(L)))


def tda_token_scores(L, dtype, A, B, N, R, n_q, ld_R, out, ld_q_out, beta=0.0, ws=None, ws_bytes=0, stream=None):
    _check(load().tda_token_scores(ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(R), n_q, ld_R, _ptr(out),
                                   ld_q_out, beta, _ptr(ws), ws_bytes, _stream(stream)))


def tda_mask_gather(L, dtype, A, B, N, rows, cols, n_coords, out, ld_out, stream=None):
    _check(load().tda_mask_gather(ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(rows), _ptr(cols), n_coords,
                                  _ptr(out), ld_out, _stream(stream)))


def tda_kfac_state_bytes(k_in, k_out) -> int:
    return int(load().tda_kfac_state_bytes(k_in, k_out))


def tda_kfac_workspace_size(L, dtype) -> int:
    return int(load().tda_kfac_workspace_size(ctypes.byref(L), dtype))


def tda_kfac_reset(k_in, k_out, state, stream=None, n_layers=1):
    _check(load().tda_kfac_reset(n_layers, k_in, k_out, _ptr(state), _stream(stream)))


def tda_kfac_accumulate_factors(L, dtype, A, B, N, state, ws, ws_bytes, stream=None):
    _check(load().tda_kfac_accumulate_factors(ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(state), _ptr(ws),
                                              ws_bytes, _stream(stream)))


def tda_project_kfac(L, dtype, A, B, N, phi, ld_phi, state, ws, ws_bytes, stream=None):
    _check(load().tda_project_kfac(ctypes.byref(L), dtype, _ptr(A), _ptr(B), N, _ptr(phi), ld_phi, _ptr(state),
                                   _ptr(ws), ws_bytes, _stream(stream)))


def tda_kfac_eigen(k_in, k_out, state, stream=None, n_layers=1):
    _check(load().tda_kfac_eigen(n_layers, k_in, k_out, _ptr(state), _stream(stream)))


def tda_kfac_accumulate_eigenvalues(k_in, k_out, state, phi, n, ld_phi, ws, ws_bytes, stream=None, n_layers=1):
    _check(load().tda_kfac_accumulate_eigenvalues(n_layers, k_in, k_out, _ptr(state), _ptr(phi), n, ld_phi, _ptr(ws),
                                                  ws_bytes, _stream(stream)))


def tda_kfac_apply(kind, k_in, k_out, state, lambda_abs, lambda_rel, q, n_q, ld_q, qhat, ld_qhat, stream=None,
                   n_layers=1):
    _check(load().tda_kfac_apply(kind, n_layers, k_in, k_out, _ptr(state), float(lambda_abs), float(lambda_rel),
                                 _ptr(q), n_q, ld_q, _ptr(qhat), ld_qhat, _stream(stream)))


def tda_precondition_state_bytes(D, state_dtype) -> int:
    return int(load().tda_precondition_state_bytes(D, state_dtype))


def tda_precondition(op, n_layers, D, state_dtype, state, phi=None, n=0, ld_phi=0, n_total=0, lambda_abs=0.0,
                     lambda_rel_mean_eig=0.0, q=None, n_q=0, ld_q=0, qhat=None, ld_qhat=0, stream=None):
    _check(load().tda_precondition(op, n_layers, D, state_dtype, _ptr(state), _ptr(phi), n, ld_phi, n_total,
                                   lambda_abs, lambda_rel_mean_eig, _ptr(q), n_q, ld_q, _ptr(qhat),
                                   ld_qhat, _stream(stream)))


def tda_precondition_info(n_layers, D, state_dtype, state, stream=None) -> list[float]:
    info = (ctypes.c_double * (4 * n_layers))()
    _check(load().tda_precondition_info(n_layers, D, state_dtype, _ptr(state), info, _stream(stream)))
    return list(info)


def tda_score(Qhat, q_dtype, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta=0.0, stream=None):
    _check(load().tda_score(_ptr(Qhat), q_dtype, n_q, ld_q, _ptr(Phi), n_t, ld_phi, D, _ptr(S), ld_S,
                            beta, _stream(stream)))


def tda_similarity_gram_engine(L, dtype, Aq, Bq, At, Bt) -> int:
    return int(load().tda_similarity_gram_engine(ctypes.byref(L), dtype, _ptr(Aq), _ptr(Bq), _ptr(At), _ptr(Bt)))


def tda_score_engine(Qhat, q_dtype, n_q, ld_q, Phi, n_t, ld_phi, D) -> int:
    return int(load().tda_score_engine(_ptr(Qhat), q_dtype, n_q, ld_q, _ptr(Phi), n_t, ld_phi, D))


def tda_topk(S, n_q, n_t, ld_S, k, idx, val=None, stream=None):
    _check(load().tda_topk(_ptr(S), n_q, n_t, ld_S, k, _ptr(idx), _ptr(val), _stream(stream)))


def tda_route(L, op, n1, n2, dtype) -> tuple[int, list[float]]:
    chosen = ctypes.c_int32(0)
    cost = (ctypes.c_double * 3)()
    _check(load().tda_route(ctypes.byref(L), op, n1, n2, dtype, ctypes.byref(chosen), cost))
    return int(chosen.value), list(cost)


def tda_route_calibrate(ws, ws_bytes, stream=None) -> list[float]:
    rates = (ctypes.c_double * 7)()
    _check(load().tda_route_calibrate(_ptr(ws), ws_bytes, _stream(stream), rates))
    return list(rates)


def tda_route_set_model(model: int) -> None:
    _check(load().tda_route_set_model(model))


def tda_selftest_bounded_wait(timeout_ns, stream=None) -> None:
    _check(load().tda_selftest_bounded_wait(timeout_ns, _stream(stream)))


def tda_device_status(stream=None) -> None:
    _check(load().tda_device_status(_stream(stream)))
