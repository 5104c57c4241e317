"""Thin ctypes binding of the C ABI in include/fiona.h (argument marshalling
only: every step of the evaluation runs in libfiona.so's CUDA kernels).

Buffers are passed as torch tensors (their ``data_ptr()``; int64 storage is
read as uint64 residues) or as raw integer addresses.  The library must have
been built (``paper_2609_35352_gb300.build.build()``); importing this module
without it raises, there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Any, Dict, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libfiona.so")
WORKLOAD_LIB_PATH = os.path.join(_HERE, "_build", "libfiona_workload.so")

FIONA_OK = 0
FIONA_ERR_ARG = -1
FIONA_ERR_MODULUS = -2
FIONA_ERR_PLAN = -3
FIONA_ERR_NOMEM = -4
FIONA_ERR_CUDA = -5
FIONA_ERR_RANGE = -6
FIONA_ERR_NODEVICE = -7
FIONA_ERR_TIMEOUT = -8
FIONA_ERR_INTERNAL = -9
FIONA_DEVICE_NONE = -1
FIONA_RESCALE_ROUND = 1
FIONA_KERNEL_AUTO = 0
FIONA_KERNEL_DIRECT = 1
FIONA_KERNEL_TILED = 2
KERNELS = {"auto": FIONA_KERNEL_AUTO, "direct": FIONA_KERNEL_DIRECT, "tiled": FIONA_KERNEL_TILED}

EXPORTED = ("fiona_ctx_create", "fiona_ctx_destroy", "fiona_plan_create", "fiona_plan_create_classes",
            "fiona_plan_destroy",
            "fiona_plan_stats", "fiona_linear_eval", "fiona_linear_eval_host", "fiona_linear_eval_host_async",
            "fiona_linear_eval_host_join",
            "fiona_check_residues", "fiona_status_str", "fiona_last_error", "fiona_abi_version",
            "fiona_plan_select_kernel", "fiona_device_check", "fiona_linear_eval_static",
            "fiona_linear_eval_level", "fiona_plan_compile", "fiona_rescale",
            "fiona_linear_eval_rescale", "fiona_ckks_embed", "fiona_encode_coeffs", "fiona_encode")
STATIC_AREA_BYTES = 1 << 20


FIONA_COMPILE_SHARE = 1
FIONA_COMPILE_SHARE_EXACT = 2
ROUTE_DTYPE = np.dtype([("kind", "i1"), ("sign", "i1"), ("reserved", "<u2"), ("pt", "<u4")])
assert ROUTE_DTYPE.itemsize == 8


class FionaError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__("%s failed: %s (%d): %s" % (where, status_str(status), status, detail))
        self.status = status


class PlanStats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_uint64) for n in (
        "n_terms", "n_nonzero_terms", "n_raw_terms", "n_signed_terms", "n_skipped_terms",
        "n_scale_groups_used", "n_nodes", "n_uses", "pmult_per_term", "pmult_grouped",
        "addsub_flat", "addsub_shared", "rescale_separate", "rescale_combined",
        "n_inputs_used", "n_plaintexts_used", "bytes_min", "wide_products")] + \
        [(n, ctypes.c_uint32) for n in (
            "N", "L", "n_in", "n_out", "n_pt", "n_groups", "tile_coeffs", "warps_per_cta",
            "smem_bytes", "ctas_per_sm", "kernel", "nodes_materialized", "addsub_executed",
                  "tensor_core_sums", "source_offsets", "const_raw_all")]

    def as_dict(self) -> Dict[str, int]:
        return {n: int(getattr(self, n)) for n, _ in self._fields_ if n != "reserved"}


_lib: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libfiona.so is not built (%s); run "
                               "paper_2609_35352_gb300.build.build()" % LIB_PATH)
        L = ctypes.CDLL(LIB_PATH)
        p, u32, i32 = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_int
        L.fiona_ctx_create.argtypes = [u32, p, u32, i32, ctypes.POINTER(p)]
        L.fiona_ctx_create.restype = i32
        L.fiona_ctx_destroy.argtypes = [p]
        L.fiona_ctx_destroy.restype = None
        L.fiona_plan_create.argtypes = [p, u32, u32, u32, p, p, u32, p, p, u32, p, p, u32, p,
                                        ctypes.POINTER(p)]
        L.fiona_plan_create.restype = i32
        L.fiona_plan_create_classes.argtypes = [p, u32, u32, u32, p, p, u32, p, p, u32, p, p, u32, p, u32, p, p]
        L.fiona_plan_create_classes.restype = i32
        L.fiona_plan_destroy.argtypes = [p]
        L.fiona_plan_destroy.restype = None
        L.fiona_plan_stats.argtypes = [p, ctypes.POINTER(PlanStats)]
        L.fiona_plan_stats.restype = i32
        L.fiona_linear_eval.argtypes = [p, p, p, p, p]
        L.fiona_linear_eval.restype = i32
        L.fiona_linear_eval_host.argtypes = [p, p, p, p, p, p, p]
        L.fiona_linear_eval_host.restype = i32
        L.fiona_linear_eval_host_async.argtypes = [p, p, p, p, p, p, p]
        L.fiona_linear_eval_host_async.restype = i32
        L.fiona_linear_eval_host_join.argtypes = [p, p]
        L.fiona_linear_eval_host_join.restype = i32
        L.fiona_check_residues.argtypes = [p, p, p, ctypes.c_uint64]
        L.fiona_check_residues.restype = i32
        L.fiona_status_str.argtypes = [i32]
        L.fiona_status_str.restype = ctypes.c_char_p
        L.fiona_last_error.argtypes = []
        L.fiona_last_error.restype = ctypes.c_char_p
        L.fiona_abi_version.argtypes = []
        L.fiona_abi_version.restype = i32
        L.fiona_plan_select_kernel.argtypes = [p, i32]
        L.fiona_plan_select_kernel.restype = i32
        L.fiona_device_check.argtypes = [p, p]
        L.fiona_device_check.restype = i32
        L.fiona_linear_eval_static.argtypes = [p, p, p, p, p]
        L.fiona_linear_eval_level.argtypes = [p, p, u32, p, p, p]
        L.fiona_linear_eval_level.restype = i32
        L.fiona_rescale.argtypes = [p, p, u32, ctypes.c_uint64, p, p, u32]
        L.fiona_rescale.restype = i32
        L.fiona_linear_eval_rescale.argtypes = [p, p, u32, p, p, p, p, u32]
        L.fiona_linear_eval_rescale.restype = i32
        L.fiona_ckks_embed.argtypes = [p, p, ctypes.c_uint64, p, ctypes.c_double, p, p]
        L.fiona_ckks_embed.restype = i32
        L.fiona_encode_coeffs.argtypes = [p, p, u32, ctypes.c_uint64, p, p]
        L.fiona_encode_coeffs.restype = i32
        L.fiona_encode.argtypes = [p, p, u32, ctypes.c_uint64, p, ctypes.c_double, p, p, p]
        L.fiona_encode.restype = i32
        L.fiona_plan_compile.argtypes = [u32, u32, u32, p, u32, p, p, p, p, p, p, p, p, p, p]
        L.fiona_plan_compile.restype = i32
        L.fiona_linear_eval_static.restype = i32
        _lib = L
    return _lib


def status_str(status: int) -> str:
    return lib().fiona_status_str(status).decode()


def last_error() -> str:
    return lib().fiona_last_error().decode()


def _check(status: int, where: str) -> None:
    if status != FIONA_OK:
        raise FionaError(status, where, last_error())


def addr(x: Any) -> int:
    """Device or host address of a torch tensor, numpy array or integer."""
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return int(x.data_ptr())
    if isinstance(x, np.ndarray):
        return int(x.ctypes.data)
    raise TypeError("cannot take the address of %r" % type(x))


def stream_handle(stream: Any) -> int:
    if stream is None:
        return 0
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


class Context:
    """fiona_ctx: ring dimension N and RNS moduli on one device."""

    def __init__(self, N: int, moduli, device: int = 0):
        q = np.ascontiguousarray(np.asarray(moduli, dtype=np.uint64))
        self._q = q
        h = ctypes.c_void_p()
        _check(lib().fiona_ctx_create(N, q.ctypes.data, q.shape[0], device, ctypes.byref(h)),
               "fiona_ctx_create")
        self.handle = h
        self.N, self.L, self.device = N, int(q.shape[0]), device

    def check_residues(self, data, count: int, stream=None) -> int:
        """FIONA_OK or FIONA_ERR_RANGE (raises on other errors)."""
        rc = lib().fiona_check_residues(self.handle, stream_handle(stream), addr(data), count)
        if rc not in (FIONA_OK, FIONA_ERR_RANGE):
            _check(rc, "fiona_check_residues")
        return rc

    def device_check(self, stream=None) -> int:
        """fiona_device_check: FIONA_OK, FIONA_ERR_TIMEOUT if a kernel gave up
        a bounded wait, or FIONA_ERR_RANGE if an encoding met a coefficient out
        of range, since the last check (raises on other errors)."""
        rc = lib().fiona_device_check(self.handle, stream_handle(stream))
        if rc not in (FIONA_OK, FIONA_ERR_TIMEOUT, FIONA_ERR_RANGE):
            _check(rc, "fiona_device_check")
        return rc

    def rescale(self, L_cur, count, polys, out, stream=None, round=False) -> None:
        """fiona_rescale: divide `count` polys ([count][L_cur][N], NTT form)
        by q_{L_cur-1} into out ([count][L_cur-1][N]), the quotient rounded
        down (or to nearest with round=True); the last limb of each input
        poly is overwritten."""
        _check(self.rescale_status(L_cur, count, polys, out, stream, round), "fiona_rescale")

    def rescale_status(self, L_cur, count, polys, out, stream=None, round=False, flags=None) -> int:
        f = (FIONA_RESCALE_ROUND if round else 0) if flags is None else int(flags)
        return lib().fiona_rescale(self.handle, stream_handle(stream), int(L_cur), int(count), addr(polys),
                                   addr(out), f)

    def ckks_embed_status(self, count, slots, scale, coeffs, work, stream=None) -> int:
        """fiona_ckks_embed: slots [count][N/2][2] float64 -> coeffs [count][N]
        int64 (work: count * N * 8 bytes)."""
        return lib().fiona_ckks_embed(self.handle, stream_handle(stream), int(count), addr(slots), float(scale),
                                      addr(coeffs), addr(work))

    def ckks_embed(self, count, slots, scale, coeffs, work, stream=None) -> None:
        _check(self.ckks_embed_status(count, slots, scale, coeffs, work, stream), "fiona_ckks_embed")

    def encode_coeffs_status(self, L_cur, count, coeffs, out, stream=None) -> int:
        """fiona_encode_coeffs: int64 coeffs [count][N] -> out [count][L_cur][N]."""
        return lib().fiona_encode_coeffs(self.handle, stream_handle(stream), int(L_cur), int(count), addr(coeffs),
                                         addr(out))

    def encode_coeffs(self, L_cur, count, coeffs, out, stream=None) -> None:
        _check(self.encode_coeffs_status(L_cur, count, coeffs, out, stream), "fiona_encode_coeffs")

    def encode_status(self, L_cur, count, slots, scale, coeffs, work, out, stream=None) -> int:
        return lib().fiona_encode(self.handle, stream_handle(stream), int(L_cur), int(count), addr(slots),
                                  float(scale), addr(coeffs), addr(work), addr(out))

    def encode(self, L_cur, count, slots, scale, coeffs, work, out, stream=None) -> None:
        """fiona_encode: slots -> RNS NTT plaintexts [count][L_cur][N]."""
        _check(self.encode_status(L_cur, count, slots, scale, coeffs, work, out, stream), "fiona_encode")

    def close(self) -> None:
        if getattr(self, "handle", None):
            lib().fiona_ctx_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _arr(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


class Plan:
    """fiona_plan: one validated, lowered layer.  ``desc`` provides n_in,
    n_out, n_pt, term_offsets, terms, group_scale_pt, group_output,
    node_offsets, children and uses (see workloads.Plan)."""

    def __init__(self, ctx: Context, desc, pt_class=None, n_class: int = 1):
        """With pt_class (a scale class per plaintext, < n_class): the plan of
        fiona_plan_create_classes, whose n_out * n_class results are laid out
        [n_out][n_class][2][L][N]."""
        self.ctx = ctx
        self._keep = []

        def ptr(a):
            self._keep.append(a)
            return a.ctypes.data if a.size else None

        offs = _arr(desc.term_offsets, np.uint32)
        terms = np.ascontiguousarray(desc.terms)
        gsp = _arr(desc.group_scale_pt, np.uint32)
        gout = _arr(desc.group_output, np.uint32)
        noffs = _arr(desc.node_offsets, np.uint32)
        ch = np.ascontiguousarray(desc.children)
        us = np.ascontiguousarray(desc.uses)
        n_nodes = max(int(noffs.shape[0]) - 1, 0)
        h = ctypes.c_void_p()
        if pt_class is None:
            rc = lib().fiona_plan_create(ctx.handle, desc.n_in, desc.n_out, desc.n_pt, ptr(offs),
                                         ptr(terms), int(gsp.shape[0]), ptr(gsp), ptr(gout),
                                         n_nodes, ptr(noffs) if n_nodes else None, ptr(ch),
                                         int(us.shape[0]), ptr(us), ctypes.byref(h))
            where = "fiona_plan_create"
        else:
            cls = _arr(pt_class, np.uint8)
            rc = lib().fiona_plan_create_classes(ctx.handle, desc.n_in, desc.n_out, desc.n_pt, ptr(offs),
                                                 ptr(terms), int(gsp.shape[0]), ptr(gsp), ptr(gout),
                                                 n_nodes, ptr(noffs) if n_nodes else None, ptr(ch),
                                                 int(us.shape[0]), ptr(us), int(n_class), ptr(cls),
                                                 ctypes.byref(h))
            where = "fiona_plan_create_classes"
        self._keep = []
        _check(rc, where)
        self.handle = h
        self.n_in, self.n_pt = desc.n_in, desc.n_pt
        self.n_out = desc.n_out * (1 if pt_class is None else int(n_class))

    def stats(self) -> Dict[str, int]:
        s = PlanStats()
        _check(lib().fiona_plan_stats(self.handle, ctypes.byref(s)), "fiona_plan_stats")
        return s.as_dict()

    def select_kernel(self, kernel) -> None:
        """Use kernel variant "auto", "direct" or "tiled" (or its FIONA_KERNEL_* value)."""
        k = KERNELS[kernel] if isinstance(kernel, str) else int(kernel)
        _check(lib().fiona_plan_select_kernel(self.handle, k), "fiona_plan_select_kernel")

    def eval(self, inputs, plaintexts, outputs, stream=None) -> None:
        """Enqueue fiona_linear_eval on `stream` (device buffers)."""
        _check(lib().fiona_linear_eval(self.handle, stream_handle(stream), addr(inputs),
                                       addr(plaintexts), addr(outputs)), "fiona_linear_eval")

    def eval_status(self, inputs, plaintexts, outputs, stream=None) -> int:
        return lib().fiona_linear_eval(self.handle, stream_handle(stream), addr(inputs),
                                       addr(plaintexts), addr(outputs))

    def eval_level(self, L_eval, inputs, plaintexts, outputs, stream=None) -> None:
        """fiona_linear_eval_level: buffers holding the first L_eval limbs."""
        _check(lib().fiona_linear_eval_level(self.handle, stream_handle(stream), int(L_eval), addr(inputs),
                                             addr(plaintexts), addr(outputs)), "fiona_linear_eval_level")

    def eval_level_status(self, L_eval, inputs, plaintexts, outputs, stream=None) -> int:
        return lib().fiona_linear_eval_level(self.handle, stream_handle(stream), int(L_eval), addr(inputs),
                                             addr(plaintexts), addr(outputs))

    def eval_rescale(self, L_eval, inputs, plaintexts, work, outputs, stream=None, round=False) -> None:
        """fiona_linear_eval_rescale: the layer at level L_eval into `work`,
        then its rescale into `outputs` ([n_out][2][L_eval-1][N])."""
        _check(self.eval_rescale_status(L_eval, inputs, plaintexts, work, outputs, stream, round),
               "fiona_linear_eval_rescale")

    def eval_rescale_status(self, L_eval, inputs, plaintexts, work, outputs, stream=None, round=False) -> int:
        return lib().fiona_linear_eval_rescale(self.handle, stream_handle(stream), int(L_eval), addr(inputs),
                                               addr(plaintexts), addr(work), addr(outputs),
                                               FIONA_RESCALE_ROUND if round else 0)

    def eval_static(self, inputs, plaintexts, outputs, stream=None) -> int:
        """fiona_linear_eval_static: no device allocation (returns the status)."""
        return lib().fiona_linear_eval_static(self.handle, stream_handle(stream), addr(inputs),
                                              addr(plaintexts), addr(outputs))

    def eval_host(self, h_inputs, d_plaintexts, h_outputs, d_inputs, d_outputs,
                  stream=None) -> None:
        """fiona_linear_eval_host: host inputs -> host outputs (synchronous)."""
        _check(lib().fiona_linear_eval_host(self.handle, stream_handle(stream), addr(h_inputs),
                                            addr(d_plaintexts), addr(h_outputs), addr(d_inputs),
                                            addr(d_outputs)), "fiona_linear_eval_host")

    def eval_host_async(self, h_inputs, d_plaintexts, h_outputs, d_inputs, d_outputs,
                        stream=None) -> None:
        """fiona_linear_eval_host_async: queued only; the result is in
        h_outputs once `stream` has completed after eval_host_join."""
        _check(lib().fiona_linear_eval_host_async(self.handle, stream_handle(stream), addr(h_inputs),
                                                  addr(d_plaintexts), addr(h_outputs), addr(d_inputs),
                                                  addr(d_outputs)), "fiona_linear_eval_host_async")

    def eval_host_join(self, stream=None) -> None:
        """fiona_linear_eval_host_join: `stream` waits for the queued output copies."""
        _check(lib().fiona_linear_eval_host_join(self.handle, stream_handle(stream)), "fiona_linear_eval_host_join")

    def close(self) -> None:
        if getattr(self, "handle", None):
            lib().fiona_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# -- device filler for synthetic inputs (libfiona_workload.so) ---------------
_wlib: Optional[ctypes.CDLL] = None


def workload_lib() -> ctypes.CDLL:
    global _wlib
    if _wlib is None:
        if not os.path.exists(WORKLOAD_LIB_PATH):
            raise RuntimeError("libfiona_workload.so is not built")
        W = ctypes.CDLL(WORKLOAD_LIB_PATH)
        W.fiona_workload_fill.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint64,
                                          ctypes.c_uint32, ctypes.c_uint32, ctypes.c_void_p,
                                          ctypes.c_uint64, ctypes.c_int]
        W.fiona_workload_fill.restype = ctypes.c_int
        W.fiona_mul_roof.argtypes = [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]
        W.fiona_mul_roof.restype = ctypes.c_int
        W.fiona_bfly_roof.argtypes = [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]
        W.fiona_bfly_roof.restype = ctypes.c_int
        _wlib = W
    return _wlib


def device_fill(dst, outer: int, L: int, N: int, moduli, key: int, mode: int = 0,
                stream=None) -> None:
    q = _arr(moduli, np.uint64)
    rc = workload_lib().fiona_workload_fill(stream_handle(stream), addr(dst), outer, L, N,
                                            q.ctypes.data, key, mode)
    if rc != 0:
        raise RuntimeError("fiona_workload_fill failed (%d)" % rc)


def mul_roof() -> Dict[str, float]:
    """fiona_mul_roof: the measured products per second of the narrow
    (radix-2^26 Karatsuba) and wide (64x64 -> 128) product-accumulates on the
    current device."""
    n, w = ctypes.c_double(), ctypes.c_double()
    rc = workload_lib().fiona_mul_roof(ctypes.byref(n), ctypes.byref(w))
    if rc != 0:
        raise RuntimeError("fiona_mul_roof failed (%d)" % rc)
    return {"narrow": n.value, "wide": w.value}


def bfly_roof() -> Dict[str, float]:
    """fiona_bfly_roof: the measured forward NTT butterflies per second of the
    rescale's butterfly, fast (moduli below 2^56) and general."""
    f, g = ctypes.c_double(), ctypes.c_double()
    rc = workload_lib().fiona_bfly_roof(ctypes.byref(f), ctypes.byref(g))
    if rc != 0:
        raise RuntimeError("fiona_bfly_roof failed (%d)" % rc)
    return {"fast": f.value, "general": g.value}


# -- host plan compiler -------------------------------------------------------
def compile_plan(n_in: int, n_out: int, n_pt: int, routes: np.ndarray, share: bool = True,
                 exact: bool = False):
    """fiona_plan_compile: the dense route matrix ``routes`` (ROUTE_DTYPE,
    shape [n_out][n_in]) to a plan description (workloads.Plan) for
    ``Plan(ctx, desc)``: terms, scale groups and, with ``share``, shared
    signed sums (``exact``: accept by the exact Add/Sub saving)."""
    from . import workloads as W
    r = np.ascontiguousarray(routes, dtype=ROUTE_DTYPE).reshape(-1)
    if r.shape[0] != n_in * n_out:
        raise ValueError("routes must hold n_out * n_in entries")
    cap = max(n_in * n_out, 1)
    offs = np.zeros(n_out + 1, np.uint32)
    terms = np.zeros(cap, W.TERM_DTYPE)
    gsp = np.zeros(cap, np.uint32)
    gout = np.zeros(cap, np.uint32)
    noffs = np.zeros(cap + 1, np.uint32)
    ch = np.zeros(cap, W.CHILD_DTYPE)
    us = np.zeros(cap, W.USE_DTYPE)
    ng, nn, nu = ctypes.c_uint32(), ctypes.c_uint32(), ctypes.c_uint32()
    flags = (FIONA_COMPILE_SHARE if share else 0) | (FIONA_COMPILE_SHARE_EXACT if share and exact else 0)
    _check(lib().fiona_plan_compile(n_in, n_out, n_pt, r.ctypes.data if r.size else None, flags,
                                    offs.ctypes.data, terms.ctypes.data, ctypes.byref(ng), gsp.ctypes.data,
                                    gout.ctypes.data, ctypes.byref(nn), noffs.ctypes.data, ch.ctypes.data,
                                    ctypes.byref(nu), us.ctypes.data), "fiona_plan_compile")
    n_terms = int(offs[n_out])
    return W.Plan(n_in=n_in, n_out=n_out, n_pt=n_pt, term_offsets=offs, terms=terms[:n_terms].copy(),
                  group_scale_pt=gsp[:ng.value].copy(), group_output=gout[:ng.value].copy(),
                  node_offsets=noffs[:nn.value + 1].copy(), children=ch[:int(noffs[nn.value])].copy(),
                  uses=us[:nu.value].copy())
