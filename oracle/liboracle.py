"""Build and call oracle.c through ctypes (test infrastructure only)."""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SRCS = [_SRC, os.path.join(_HERE, "rescale.c"), os.path.join(_HERE, "encode.c")]
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "liboracle.so")
_handle: Optional[ctypes.CDLL] = None


def build(force: bool = False) -> str:
    """Compile oracle.c with the host C compiler (plain -O2, no tuning)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or any(os.path.getmtime(_LIB) < os.path.getmtime(f) for f in _SRCS):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp] + _SRCS + ["-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _setup(lib: ctypes.CDLL) -> ctypes.CDLL:
    p = ctypes.c_void_p
    u32, u64 = ctypes.c_uint32, ctypes.c_uint64
    lib.oracle_linear_eval.argtypes = [u64, u32, p, u32, u32, u32, p, p, p, p, p, p,
                                       u32, p, p, p, p]
    lib.oracle_linear_eval.restype = ctypes.c_int
    lib.oracle_linear_eval_classes.argtypes = [u64, u32, p, u32, u32, u32, p, p, p, p, p, p,
                                               u32, p, u32, p, p, p, p]
    lib.oracle_linear_eval_dag.argtypes = [u64, u32, p, u32, u32, u32, p, p, p, p, p, p,
                                           u32, p, u32, p, p, p, p, u32, p, p, p, p,
                                           p, p, p]
    lib.oracle_linear_eval_dag.restype = ctypes.c_int
    if hasattr(lib, "oracle_rescale"):
        lib.oracle_min_root.argtypes = [u64, u32]
        lib.oracle_min_root.restype = u64
        for f in ("oracle_ntt_direct", "oracle_intt_direct"):
            getattr(lib, f).argtypes = [p, p, u32, u64, u64]
            getattr(lib, f).restype = None
        for f in ("oracle_ntt_fast", "oracle_intt_fast"):
            getattr(lib, f).argtypes = [p, u32, u64, u64]
            getattr(lib, f).restype = None
        lib.oracle_rescale.argtypes = [u64, u32, u32, p, p, p, ctypes.c_int, ctypes.c_int]
        lib.oracle_rescale.restype = ctypes.c_int
    if hasattr(lib, "oracle_ckks_embed"):
        lib.oracle_ckks_embed.argtypes = [u32, p, ctypes.c_double, p, u32, p]
        lib.oracle_ckks_embed.restype = ctypes.c_int
        lib.oracle_encode_coeffs.argtypes = [u32, u32, p, u64, p, p, ctypes.c_int]
        lib.oracle_encode_coeffs.restype = ctypes.c_int
    return lib


def load() -> ctypes.CDLL:
    global _handle
    if _handle is None:
        _handle = _setup(ctypes.CDLL(build()))
    return _handle


def load_variant(src_path: str, out_path: str) -> ctypes.CDLL:
    """Compile and load another copy of the oracle source (used by the test
    that plants mistakes in a copy of the oracle to show the pins catch them)."""
    subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", out_path, src_path],
                   check=True)
    return _setup(ctypes.CDLL(out_path))


def _ptr(a: np.ndarray) -> ctypes.c_void_p:
    return ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def _term_arrays(plan):
    t = plan.terms
    return (_c(plan.term_offsets, np.uint32), _c(t["input"], np.uint32), _c(t["kind"], np.int8),
            _c(t["sign"], np.int8), _c(t["pt"], np.uint32), _c(t["group"], np.uint32),
            _c(plan.group_scale_pt, np.uint32))


def linear_eval(plan, moduli, inputs: np.ndarray, plaintexts: np.ndarray,
                lib: Optional[ctypes.CDLL] = None) -> np.ndarray:
    """Flat-form evaluation.  inputs [n_in][2][L][n], plaintexts [n_pt][L][n]
    (uint64); returns outputs [n_out][2][L][n]."""
    lib = lib or load()
    q = _c(moduli, np.uint64)
    L = q.shape[0]
    inputs = _c(inputs, np.uint64)
    plaintexts = _c(plaintexts, np.uint64)
    n = inputs.shape[-1] if inputs.ndim == 4 else plaintexts.shape[-1]
    assert inputs.shape == (plan.n_in, 2, L, n), inputs.shape
    assert plaintexts.shape == (plan.n_pt, L, n), plaintexts.shape
    out = np.zeros((plan.n_out, 2, L, n), dtype=np.uint64)
    arrs = _term_arrays(plan)
    rc = lib.oracle_linear_eval(n, L, _ptr(q), plan.n_in, plan.n_out, plan.n_pt,
                                *[_ptr(a) for a in arrs[:6]], plan.n_groups, _ptr(arrs[6]),
                                _ptr(inputs), _ptr(plaintexts), _ptr(out))
    if rc != 0:
        raise ValueError("oracle rejected the plan")
    return out


def linear_eval_classes(plan, moduli, pt_class, n_class: int, inputs: np.ndarray, plaintexts: np.ndarray,
                        lib: Optional[ctypes.CDLL] = None) -> np.ndarray:
    """Evaluation with plaintext scale classes: returns [n_out][n_class][2][L][n],
    output j's terms of class s (by their plaintext) in [j][s]."""
    lib = lib or load()
    q = _c(moduli, np.uint64)
    L = q.shape[0]
    inputs = _c(inputs, np.uint64)
    plaintexts = _c(plaintexts, np.uint64)
    n = inputs.shape[-1] if inputs.ndim == 4 else plaintexts.shape[-1]
    assert inputs.shape == (plan.n_in, 2, L, n), inputs.shape
    assert plaintexts.shape == (plan.n_pt, L, n), plaintexts.shape
    cls = _c(pt_class, np.uint8)
    assert cls.shape == (plan.n_pt,)
    out = np.zeros((plan.n_out, n_class, 2, L, n), dtype=np.uint64)
    arrs = _term_arrays(plan)
    rc = lib.oracle_linear_eval_classes(n, L, _ptr(q), plan.n_in, plan.n_out, plan.n_pt,
                                        *[_ptr(a) for a in arrs[:6]], plan.n_groups, _ptr(arrs[6]),
                                        n_class, _ptr(cls), _ptr(inputs), _ptr(plaintexts), _ptr(out))
    if rc != 0:
        raise ValueError("oracle rejected the plan or its classes")
    return out


def linear_eval_dag(plan, moduli, inputs: np.ndarray, plaintexts: np.ndarray,
                    lib: Optional[ctypes.CDLL] = None) -> np.ndarray:
    """DAG-form evaluation: each shared signed sum formed once, then used."""
    lib = lib or load()
    q = _c(moduli, np.uint64)
    L = q.shape[0]
    inputs = _c(inputs, np.uint64)
    plaintexts = _c(plaintexts, np.uint64)
    n = inputs.shape[-1]
    assert inputs.shape == (plan.n_in, 2, L, n)
    assert plaintexts.shape == (plan.n_pt, L, n)
    out = np.zeros((plan.n_out, 2, L, n), dtype=np.uint64)
    arrs = _term_arrays(plan)
    ch = plan.children
    us = plan.uses
    dag = (_c(plan.node_offsets, np.uint32), _c(ch["ref"], np.uint32), _c(ch["is_node"], np.int8),
           _c(ch["sign"], np.int8))
    ua = (_c(us["output"], np.uint32), _c(us["group"], np.uint32), _c(us["node"], np.uint32),
          _c(us["sign"], np.int8))
    rc = lib.oracle_linear_eval_dag(n, L, _ptr(q), plan.n_in, plan.n_out, plan.n_pt,
                                    *[_ptr(a) for a in arrs[:6]], plan.n_groups, _ptr(arrs[6]),
                                    plan.n_nodes, *[_ptr(a) for a in dag],
                                    plan.n_uses, *[_ptr(a) for a in ua],
                                    _ptr(inputs), _ptr(plaintexts), _ptr(out))
    if rc != 0:
        raise ValueError("oracle rejected the plan or its DAG")
    return out


# -- rescale (rescale.c) --------------------------------------------------------
def min_root(q: int, N: int) -> int:
    """The least primitive 2N-th root of unity mod q."""
    return int(load().oracle_min_root(q, N))


def ntt(a: np.ndarray, q: int, fast: bool = True) -> np.ndarray:
    """Forward NTT of one length-N residue vector (bit-reversed order)."""
    a = _c(a, np.uint64)
    N = a.shape[0]
    psi = min_root(q, N)
    if fast:
        out = a.copy()
        load().oracle_ntt_fast(_ptr(out), N, q, psi)
    else:
        out = np.zeros_like(a)
        load().oracle_ntt_direct(_ptr(a), _ptr(out), N, q, psi)
    return out


def intt(A: np.ndarray, q: int, fast: bool = True) -> np.ndarray:
    A = _c(A, np.uint64)
    N = A.shape[0]
    psi = min_root(q, N)
    if fast:
        out = A.copy()
        load().oracle_intt_fast(_ptr(out), N, q, psi)
    else:
        out = np.zeros_like(A)
        load().oracle_intt_direct(_ptr(A), _ptr(out), N, q, psi)
    return out


def rescale(moduli, polys: np.ndarray, fast: bool = True, round: bool = False) -> np.ndarray:
    """Rescale polys [count][L][N] (NTT form) by the last modulus -> [count][L-1][N]
    (quotient rounded down, or to nearest with round=True)."""
    y = _c(polys, np.uint64)
    count, L, N = y.shape
    out = np.zeros((count, L - 1, N), np.uint64)
    qs = _c(list(moduli)[:L], np.uint64)
    rc = load().oracle_rescale(count, N, L, _ptr(qs), _ptr(y), _ptr(out), 1 if fast else 0, 1 if round else 0)
    if rc != 0:
        raise ValueError("oracle_rescale: arguments it cannot evaluate")
    return out


# -- plaintext encoding (encode.c) ------------------------------------------------
def ckks_embed(slots: np.ndarray, scale: float, idx=None) -> np.ndarray:
    """Integer coefficients round(scale * m_i) of the encoding of one slot
    vector (complex, length N/2), at the coefficient indices idx (all if
    None)."""
    z = np.ascontiguousarray(np.asarray(slots, dtype=np.complex128))
    n = z.shape[0]
    N = 2 * n
    zz = np.ascontiguousarray(np.stack([z.real, z.imag], axis=-1), dtype=np.float64)
    ix = _c(np.arange(N) if idx is None else idx, np.uint32)
    out = np.zeros(ix.shape[0], dtype=np.int64)
    rc = load().oracle_ckks_embed(N, _ptr(zz), float(scale), _ptr(ix), ix.shape[0], _ptr(out))
    if rc != 0:
        raise ValueError("oracle_ckks_embed: coefficient out of range or bad argument")
    return out


def encode_coeffs(moduli, coeffs: np.ndarray, fast: bool = True) -> np.ndarray:
    """Integer polys [count][N] (int64) -> NTT form [count][L][N] (uint64)."""
    c = _c(coeffs, np.int64)
    if c.ndim == 1:
        c = c.reshape(1, -1)
    count, N = c.shape
    q = _c(list(moduli), np.uint64)
    out = np.zeros((count, q.shape[0], N), np.uint64)
    rc = load().oracle_encode_coeffs(N, q.shape[0], _ptr(q), count, _ptr(c), _ptr(out), 1 if fast else 0)
    if rc != 0:
        raise ValueError("oracle_encode_coeffs: a modulus has no primitive 2N-th root")
    return out
