"""fp64 CPU oracle for the projection / routing / preconditioning / scoring path.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / reference leg of ``bench.py`` may import this package. The
product library (``paper_2609_38767_gb300``) never imports it, and it never
imports the product library.

The arithmetic lives in ``oracle.c`` (plain C, double precision); this module
only compiles it and marshals numpy arrays through ctypes. Every array passed
in is converted to a C-contiguous float64 copy first.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so next to it (gcc, OpenMP, no FMA contraction)."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "oracle.h"))
    ):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        D = ctypes.POINTER(ctypes.c_double)
        I64, U64, U32, I32 = ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int32
        sig = {
            "oracle_mix64": (U64, [U64]),
            "oracle_splitmix64_next": (U64, [ctypes.POINTER(U64)]),
            "oracle_proj_sign": (I32, [U64, U32, I32, I64, I64]),
            "oracle_proj_entries": (None, [U64, U32, I32, I32, I64, I64, ctypes.POINTER(ctypes.c_int8)]),
            "oracle_proj_matrix": (None, [U64, U32, I32, I32, I64, I64, D]),
            "oracle_materialize": (None, [I64, I64, I64, D, D, D]),
            "oracle_project_with": (None, [I64, I64, I64, I64, I64, D, D, D, D, D]),
            "oracle_project_factored": (None, [I64, I64, I64, I64, I64, I64, U64, U32, I32, D, D, D]),
            "oracle_project_materialized": (None, [I64, I64, I64, I64, I64, I64, U64, U32, I32, D, D, D]),
            "oracle_similarity_materialized": (None, [I64, I64, I64, I64, D, D, I64, D, D, D]),
            "oracle_similarity_gram": (None, [I64, I64, I64, I64, D, D, I64, D, D, D]),
            "oracle_sq_norms_materialized": (None, [I64, I64, I64, I64, D, D, D]),
            "oracle_sq_norms_gram": (None, [I64, I64, I64, I64, D, D, D]),
            "oracle_cosine": (None, [I64, I64, D, D, D, D]),
            "oracle_fisher": (None, [I64, I64, D, D]),
            "oracle_damping": (ctypes.c_double, [I64, D, ctypes.c_double, ctypes.c_double]),
            "oracle_cholesky": (I32, [I64, D]),
            "oracle_precondition": (I32, [I64, D, ctypes.c_double, I64, D, D]),
            "oracle_damping_features": (ctypes.c_double, [I64, I64, D, ctypes.c_double, ctypes.c_double]),
            "oracle_precondition_lowrank": (I32, [I64, I64, D, ctypes.c_double, I64, D, D]),
            "oracle_kfac_covariances": (None, [I64, I64, I64, I64, I64, I64, U64, U32, I32, D, D, D, D]),
            "oracle_sym_eig": (I32, [I64, D, D, D]),
            "oracle_kfac_eigenvalues": (None, [I64, I64, D, D, D]),
            "oracle_ekfac_eigenvalues": (None, [I64, I64, I64, D, D, D, D]),
            "oracle_kfac_damping": (ctypes.c_double, [I64, I64, D, ctypes.c_double, ctypes.c_double]),
            "oracle_kfac_precondition": (None, [I64, I64, D, D, D, ctypes.c_double, I64, D, D]),
            "oracle_token_scores": (None, [I64, I64, I64, I64, I64, I64, U64, U32, I32, D, D, I64, D, D]),
            "oracle_mask_gather": (None, [I64, I64, I64, I64, D, D, I64, ctypes.POINTER(I32), ctypes.POINTER(I32),
                                          D]),
            "oracle_score": (None, [I64, I64, I64, D, D, D]),
            "oracle_topk": (None, [I64, I64, D, I32, ctypes.POINTER(I32), D]),
            "oracle_route_costs": (I32, [I32, I64, I64, I64, I64, I64, I64, I64, D]),
            "oracle_set_threads": (None, [I32]),
            "oracle_get_threads": (I32, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _f64(x) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


def _p(x: np.ndarray):
    return x.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


# ---------------------------------------------------------------- hash / maps
def mix64(z: int) -> int:
    return int(_load().oracle_mix64(ctypes.c_uint64(z)))


def splitmix64_sequence(state: int, n: int) -> list[int]:
    s = ctypes.c_uint64(state)
    return [int(_load().oracle_splitmix64_next(ctypes.byref(s))) for _ in range(n)]


def proj_sign(seed: int, layer: int, side: int, r: int, c: int) -> int:
    return int(_load().oracle_proj_sign(seed, layer, side, r, c))


def proj_entries(seed: int, layer: int, side: int, rows: int, cols: int, kind: int = 0) -> np.ndarray:
    out = np.empty((rows, cols), dtype=np.int8)
    _load().oracle_proj_entries(seed, layer, side, kind, rows, cols,
                                out.ctypes.data_as(ctypes.POINTER(ctypes.c_int8)))
    return out


def proj_matrix(seed: int, layer: int, side: int, rows: int, cols: int, kind: int = 0) -> np.ndarray:
    out = np.empty((rows, cols), dtype=np.float64)
    _load().oracle_proj_matrix(seed, layer, side, kind, rows, cols, _p(out))
    return out


# ---------------------------------------------------------------- gradients
def materialize(A, B) -> np.ndarray:
    """A: (T, d_in), B: (T, d_out) -> G (d_out, d_in)."""
    A, B = _f64(A), _f64(B)
    T, d_in = A.shape
    d_out = B.shape[1]
    G = np.empty((d_out, d_in))
    _load().oracle_materialize(T, d_in, d_out, _p(A), _p(B), _p(G))
    return G


def project_with(A, B, P_in, P_out) -> np.ndarray:
    """One example with explicit maps: A (T,d_in), B (T,d_out), P_in (d_in,k_in), P_out (d_out,k_out)."""
    A, B, P_in, P_out = _f64(A), _f64(B), _f64(P_in), _f64(P_out)
    T, d_in = A.shape
    d_out = B.shape[1]
    k_in, k_out = P_in.shape[1], P_out.shape[1]
    phi = np.empty((k_out, k_in))
    _load().oracle_project_with(T, d_in, d_out, k_in, k_out, _p(P_in), _p(P_out), _p(A), _p(B), _p(phi))
    return phi


def project(A, B, k_in: int, k_out: int, seed: int, layer: int, kind: int = 0,
            route: str = "factored") -> np.ndarray:
    """A: (N,T,d_in), B: (N,T,d_out) -> Phi (N, k_out, k_in)."""
    A, B = _f64(A), _f64(B)
    N, T, d_in = A.shape
    d_out = B.shape[2]
    phi = np.empty((N, k_out, k_in))
    fn = _load().oracle_project_factored if route == "factored" else _load().oracle_project_materialized
    fn(N, T, d_in, d_out, k_in, k_out, seed, layer, kind, _p(A), _p(B), _p(phi))
    return phi


def similarity(Aq, Bq, At, Bt, route: str = "gram") -> np.ndarray:
    Aq, Bq, At, Bt = _f64(Aq), _f64(Bq), _f64(At), _f64(Bt)
    n_q, T, d_in = Aq.shape
    n_t = At.shape[0]
    d_out = Bq.shape[2]
    S = np.empty((n_q, n_t))
    fn = _load().oracle_similarity_gram if route == "gram" else _load().oracle_similarity_materialized
    fn(T, d_in, d_out, n_q, _p(Aq), _p(Bq), n_t, _p(At), _p(Bt), _p(S))
    return S


def sq_norms(A, B, route: str = "gram") -> np.ndarray:
    """Squared Frobenius norms of the N per-example gradients (N,T,d) factors."""
    A, B = _f64(A), _f64(B)
    N, T, d_in = A.shape
    d_out = B.shape[2]
    out = np.empty(N)
    fn = _load().oracle_sq_norms_gram if route == "gram" else _load().oracle_sq_norms_materialized
    fn(N, T, d_in, d_out, _p(A), _p(B), _p(out))
    return out


def cosine(S, nq, nt) -> np.ndarray:
    S, nq, nt = _f64(S), _f64(nq), _f64(nt)
    C = np.empty_like(S)
    _load().oracle_cosine(S.shape[0], S.shape[1], _p(S), _p(nq), _p(nt), _p(C))
    return C


# ---------------------------------------------------------------- preconditioning
def fisher(phi) -> np.ndarray:
    phi = _f64(phi)
    N = phi.shape[0]
    phi = phi.reshape(N, -1)
    D = phi.shape[1]
    F = np.empty((D, D))
    _load().oracle_fisher(D, N, _p(phi), _p(F))
    return F


def damping(F, lambda_abs: float, lambda_rel: float) -> float:
    F = _f64(F)
    return float(_load().oracle_damping(F.shape[0], _p(F), lambda_abs, lambda_rel))


def cholesky(M) -> tuple[np.ndarray, int]:
    L = _f64(M).copy()
    st = int(_load().oracle_cholesky(L.shape[0], _p(L)))
    return L, st


def precondition(F, lam: float, Q) -> np.ndarray:
    F, Q = _f64(F), _f64(Q)
    D = F.shape[0]
    Q = Q.reshape(-1, D)
    out = np.empty_like(Q)
    st = int(_load().oracle_precondition(D, _p(F), lam, Q.shape[0], _p(Q), _p(out)))
    if st != 0:
        raise np.linalg.LinAlgError(f"F + lambda I not positive definite (minor {st})")
    return out


def damping_features(phi, lambda_abs: float, lambda_rel: float) -> float:
    """lambda from the features (N, D) without forming F."""
    phi = _f64(phi)
    phi = phi.reshape(phi.shape[0], -1)
    return float(_load().oracle_damping_features(phi.shape[1], phi.shape[0], _p(phi), lambda_abs, lambda_rel))


def precondition_lowrank(phi, lam: float, Q) -> np.ndarray:
    """(F + lam I)^{-1} Q with F = Phi^T Phi / N given by Phi (N, D): Woodbury, an N x N solve."""
    phi, Q = _f64(phi), _f64(Q)
    N = phi.shape[0]
    phi = phi.reshape(N, -1)
    D = phi.shape[1]
    Q = Q.reshape(-1, D)
    out = np.empty_like(Q)
    st = int(_load().oracle_precondition_lowrank(D, N, _p(phi), lam, Q.shape[0], _p(Q), _p(out)))
    if st != 0:
        raise np.linalg.LinAlgError(f"N lambda I + Phi Phi^T not positive definite (minor {st})")
    return out


# ---------------------------------------------------------------- K-FAC / EK-FAC
def kfac_covariances(A, B, k_in: int, k_out: int, seed: int, layer: int, kind: int = 0):
    """A (N,T,d_in), B (N,T,d_out) -> (Ca (k_in,k_in), Cg (k_out,k_out)), token-averaged."""
    A, B = _f64(A), _f64(B)
    N, T, d_in = A.shape
    d_out = B.shape[2]
    Ca, Cg = np.empty((k_in, k_in)), np.empty((k_out, k_out))
    _load().oracle_kfac_covariances(N, T, d_in, d_out, k_in, k_out, seed, layer, kind, _p(A), _p(B),
                                    _p(Ca), _p(Cg))
    return Ca, Cg


def sym_eig(C):
    """-> (w ascending, U with eigenvectors in columns, sweeps)."""
    C = _f64(C)
    n = C.shape[0]
    w, U = np.empty(n), np.empty((n, n))
    sweeps = int(_load().oracle_sym_eig(n, _p(C), _p(w), _p(U)))
    return w, U, sweeps


def kfac_eigenvalues(wa, wg) -> np.ndarray:
    wa, wg = _f64(wa), _f64(wg)
    Lam = np.empty((wg.size, wa.size))
    _load().oracle_kfac_eigenvalues(wa.size, wg.size, _p(wa), _p(wg), _p(Lam))
    return Lam


def ekfac_eigenvalues(phi, Ua, Ug) -> np.ndarray:
    phi, Ua, Ug = _f64(phi), _f64(Ua), _f64(Ug)
    k_in, k_out = Ua.shape[0], Ug.shape[0]
    N = phi.shape[0]
    Lam = np.empty((k_out, k_in))
    _load().oracle_ekfac_eigenvalues(N, k_in, k_out, _p(phi), _p(Ua), _p(Ug), _p(Lam))
    return Lam


def kfac_damping(Lam, lambda_abs: float, lambda_rel: float) -> float:
    Lam = _f64(Lam)
    return float(_load().oracle_kfac_damping(Lam.shape[1], Lam.shape[0], _p(Lam), lambda_abs, lambda_rel))


def kfac_precondition(Ua, Ug, Lam, lam: float, Q) -> np.ndarray:
    Ua, Ug, Lam, Q = _f64(Ua), _f64(Ug), _f64(Lam), _f64(Q)
    k_in, k_out = Ua.shape[0], Ug.shape[0]
    Q = Q.reshape(-1, k_out * k_in)
    out = np.empty_like(Q)
    _load().oracle_kfac_precondition(k_in, k_out, _p(Ua), _p(Ug), _p(Lam), lam, Q.shape[0], _p(Q), _p(out))
    return out


# ---------------------------------------------------------------- token scores / masks
def token_scores(A, B, R, k_in: int, k_out: int, seed: int, layer: int, kind: int = 0) -> np.ndarray:
    """A (N,T,d_in), B (N,T,d_out), R (n_q, k_out, k_in) -> s (n_q, N, T)."""
    A, B, R = _f64(A), _f64(B), _f64(R)
    N, T, d_in = A.shape
    d_out = B.shape[2]
    n_q = R.shape[0]
    out = np.empty((n_q, N, T))
    _load().oracle_token_scores(N, T, d_in, d_out, k_in, k_out, seed, layer, kind, _p(A), _p(B), n_q, _p(R),
                                _p(out))
    return out


def mask_gather(A, B, rows, cols) -> np.ndarray:
    """DW entries at (rows[m], cols[m]) for each example: (N, n_coords)."""
    A, B = _f64(A), _f64(B)
    N, T, d_in = A.shape
    d_out = B.shape[2]
    rows = np.ascontiguousarray(rows, dtype=np.int32)
    cols = np.ascontiguousarray(cols, dtype=np.int32)
    out = np.empty((N, rows.size))
    ip = ctypes.POINTER(ctypes.c_int32)
    _load().oracle_mask_gather(N, T, d_in, d_out, _p(A), _p(B), rows.size, rows.ctypes.data_as(ip),
                               cols.ctypes.data_as(ip), _p(out))
    return out


# ---------------------------------------------------------------- scores
def score(Qhat, phi) -> np.ndarray:
    Qhat, phi = _f64(Qhat), _f64(phi)
    n_q = Qhat.shape[0]
    n_t = phi.shape[0]
    Qhat = Qhat.reshape(n_q, -1)
    phi = phi.reshape(n_t, -1)
    D = Qhat.shape[1]
    S = np.empty((n_q, n_t))
    _load().oracle_score(n_q, n_t, D, _p(Qhat), _p(phi), _p(S))
    return S


def topk(S, k: int) -> tuple[np.ndarray, np.ndarray]:
    S = _f64(S)
    n_q, n_t = S.shape
    idx = np.empty((n_q, k), dtype=np.int32)
    val = np.empty((n_q, k))
    _load().oracle_topk(n_q, n_t, _p(S), k, idx.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), _p(val))
    return idx, val


# ---------------------------------------------------------------- routing
OP_PROJECT, OP_SIM_PROJECTED, OP_SIM_EXACT, OP_NORM_PROJECTED, OP_NORM_EXACT = 0, 1, 2, 3, 4


def route_costs(op: int, n1: int, n2: int, T: int, d_in: int, d_out: int,
                k_in: int = 0, k_out: int = 0) -> tuple[int, np.ndarray]:
    cost = np.empty(3)
    best = int(_load().oracle_route_costs(op, n1, n2, T, d_in, d_out, k_in, k_out, _p(cost)))
    return best, cost


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def get_threads() -> int:
    return int(_load().oracle_get_threads())
