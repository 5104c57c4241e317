"""Build and call oracle.c through ctypes (test infrastructure only)."""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "liboracle.so")
_handle: Optional[ctypes.CDLL] = None


def build(force: bool = False) -> str:
    """Compile oracle.c with the host C compiler (plain -O2, no tuning)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC],
                       check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _setup(lib: ctypes.CDLL) -> ctypes.CDLL:
    p = ctypes.c_void_p
    u32, u64 = ctypes.c_uint32, ctypes.c_uint64
    lib.oracle_linear_eval.argtypes = [u64, u32, p, u32, u32, u32, p, p, p, p, p, p,
                                       u32, p, p, p, p]
    lib.oracle_linear_eval.restype = ctypes.c_int
    lib.oracle_linear_eval_dag.argtypes = [u64, u32, p, u32, u32, u32, p, p, p, p, p, p,
                                           u32, p, u32, p, p, p, p, u32, p, p, p, p,
                                           p, p, p]
    lib.oracle_linear_eval_dag.restype = ctypes.c_int
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
