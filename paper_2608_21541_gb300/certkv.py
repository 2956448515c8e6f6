"""Thin Python binding of the CertKV C ABI (include/certkv.h).

Argument marshalling only: every step of the compression pass and of decode
runs in the CUDA library ``libcertkv.so``.  PyTorch provides device memory and
streams.  The functions carry the C names; tensors are torch CUDA tensors in
the layouts the header documents.  If the library has not been built this
module raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass
from typing import Optional

import torch

from . import build as _build

OK, EINVAL, EBUDGET, EWORKSPACE, ECAPACITY, ECUDA, ETOOLARGE = range(7)
STATUS_NONFINITE = 1
STATUS_ZERO_TAIL = 2
STATUS_TIMEOUT = 4
STATUS_BOUNDS = 8
STAT_CENTERED, STAT_UNCENTERED, STAT_TAIL_MASS = 0, 1, 2


class certkv_shape(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("layers", ctypes.c_int32), ("hq", ctypes.c_int32),
                ("hkv", ctypes.c_int32), ("n", ctypes.c_int32), ("d", ctypes.c_int32),
                ("w", ctypes.c_int32)]


class certkv_params(ctypes.Structure):
    _fields_ = [("scale", ctypes.c_float), ("pool_kernel", ctypes.c_int32),
                ("protect_window", ctypes.c_int32), ("alpha_num", ctypes.c_int32),
                ("alpha_den", ctypes.c_int32), ("bisect_steps", ctypes.c_int32),
                ("statistic", ctypes.c_int32), ("tail_slot", ctypes.c_int32),
                ("allocator", ctypes.c_int32), ("tail_clusters", ctypes.c_int32)]


class certkv_packed(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("offsets", ctypes.c_void_p),
                ("real_counts", ctypes.c_void_p), ("positions", ctypes.c_void_p),
                ("capacity_slots", ctypes.c_int64), ("tail_f32", ctypes.c_void_p),
                ("tail_mass", ctypes.c_void_p), ("cluster_meta", ctypes.c_void_p),
                ("kept_vmax", ctypes.c_void_p)]


EXPORTED = ("certkv_default_params", "certkv_live_budget", "certkv_workspace_bytes",
            "certkv_decode_workspace_bytes", "certkv_score", "certkv_curves",
            "certkv_compress_scored", "certkv_compress", "certkv_decode_attn",
            "certkv_read_status", "certkv_strerror", "certkv_trace_enable",
            "certkv_trace_report", "certkv_decode_attn_noalloc", "certkv_host_workspace_bytes",
            "certkv_compress_host", "certkv_decode_certified", "certkv_fixed_row_workspace_bytes",
            "certkv_fixed_row_stats", "certkv_coverage_workspace_bytes",
            "certkv_coverage_profile", "certkv_sampled_workspace_bytes",
            "certkv_sampled_compensation", "certkv_compress_host_copyback",
            "certkv_workspace_guard_arm", "certkv_workspace_guard_check",
            "certkv_selftest_bounded_wait")

_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def load_library(path: Optional[str] = None):
    """Load libcertkv.so (built by ``build()``; the environment variable
    CERTKV_LIBRARY may name another build of it, such as the bounds-checking
    one); raise if it is missing."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = path or os.environ.get("CERTKV_LIBRARY") or _build.LIB
        if not os.path.exists(path):
            raise RuntimeError(
                f"CertKV CUDA library not found at {path}; build it with "
                "paper_2608_21541_gb300.build.build() (nvcc, sm_103a)")
        lib = ctypes.CDLL(path)
        P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        sp, pp, kp = (ctypes.POINTER(certkv_shape), ctypes.POINTER(certkv_params),
                      ctypes.POINTER(certkv_packed))
        lib.certkv_default_params.argtypes = [pp]
        lib.certkv_default_params.restype = None
        lib.certkv_live_budget.argtypes = [I32, I32, I64, I64]
        lib.certkv_live_budget.restype = I64
        lib.certkv_workspace_bytes.argtypes = [sp, pp]
        lib.certkv_workspace_bytes.restype = SZ
        lib.certkv_decode_workspace_bytes.argtypes = [sp]
        lib.certkv_decode_workspace_bytes.restype = SZ
        lib.certkv_score.argtypes = [sp, P, P, pp, P, P, SZ, P]
        lib.certkv_score.restype = ctypes.c_int
        lib.certkv_curves.argtypes = [sp, P, P, pp, P, P, P, SZ, P]
        lib.certkv_curves.restype = ctypes.c_int
        lib.certkv_compress_scored.argtypes = [sp, P, P, P, I64, pp, kp, P, SZ, P]
        lib.certkv_compress_scored.restype = ctypes.c_int
        lib.certkv_compress.argtypes = [sp, P, P, P, I64, pp, kp, P, SZ, P]
        lib.certkv_compress.restype = ctypes.c_int
        lib.certkv_decode_attn.argtypes = [sp, P, kp, ctypes.c_float, I32, P, P, SZ, P]
        lib.certkv_decode_attn.restype = ctypes.c_int
        lib.certkv_read_status.argtypes = [P, P]
        lib.certkv_read_status.restype = ctypes.c_int
        lib.certkv_workspace_guard_arm.argtypes = [sp, pp, P, SZ, P]
        lib.certkv_workspace_guard_arm.restype = ctypes.c_int
        lib.certkv_workspace_guard_check.argtypes = [sp, pp, P, SZ, P]
        lib.certkv_workspace_guard_check.restype = ctypes.c_int
        lib.certkv_selftest_bounded_wait.argtypes = [P]
        lib.certkv_selftest_bounded_wait.restype = ctypes.c_int
        lib.certkv_strerror.argtypes = [ctypes.c_int]
        lib.certkv_strerror.restype = ctypes.c_char_p
        lib.certkv_trace_enable.argtypes = [ctypes.c_int]
        lib.certkv_trace_enable.restype = ctypes.c_int
        lib.certkv_trace_report.argtypes = [ctypes.c_char_p, SZ]
        lib.certkv_trace_report.restype = ctypes.c_int
        lib.certkv_decode_attn_noalloc.argtypes = [sp, P, kp, ctypes.c_float, I32, P, P]
        lib.certkv_decode_attn_noalloc.restype = ctypes.c_int
        lib.certkv_host_workspace_bytes.argtypes = [sp, pp, I32]
        lib.certkv_host_workspace_bytes.restype = SZ
        lib.certkv_compress_host.argtypes = [sp, P, P, P, I64, pp, I32, kp, P, SZ, P]
        lib.certkv_compress_host.restype = ctypes.c_int
        lib.certkv_compress_host_copyback.argtypes = [sp, P, P, P, I64, pp, I32, kp, kp, P, SZ, P]
        lib.certkv_compress_host_copyback.restype = ctypes.c_int
        lib.certkv_decode_certified.argtypes = [sp, P, kp, ctypes.c_float, I32, I32, P, P, P, P,
                                                SZ, P]
        lib.certkv_decode_certified.restype = ctypes.c_int
        lib.certkv_fixed_row_workspace_bytes.argtypes = [sp]
        lib.certkv_fixed_row_workspace_bytes.restype = SZ
        lib.certkv_fixed_row_stats.argtypes = [sp, P, P, P, P, kp, ctypes.c_float, I32, P, P, SZ,
                                                    P]
        lib.certkv_fixed_row_stats.restype = ctypes.c_int
        lib.certkv_coverage_workspace_bytes.argtypes = [sp]
        lib.certkv_coverage_workspace_bytes.restype = SZ
        lib.certkv_coverage_profile.argtypes = [sp, P, P, ctypes.c_float, P, I32, P, I32, P, I32,
                                                P, P, P, P, P, P, P, SZ, P]
        lib.certkv_coverage_profile.restype = ctypes.c_int
        lib.certkv_sampled_workspace_bytes.argtypes = [sp]
        lib.certkv_sampled_workspace_bytes.restype = SZ
        lib.certkv_sampled_compensation.argtypes = [sp, P, P, P, kp, ctypes.c_float, I32, P, P, P,
                                                    P, SZ, P]
        lib.certkv_sampled_compensation.restype = ctypes.c_int
        _lib = lib
        return lib


class CertKVError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {certkv_strerror(code)} (code {code})")
        self.code = code


def _check(code: int, where: str):
    if code != OK:
        raise CertKVError(code, where)


def certkv_strerror(code: int) -> str:
    return load_library().certkv_strerror(int(code)).decode()


def certkv_default_params(**overrides) -> certkv_params:
    p = certkv_params()
    load_library().certkv_default_params(ctypes.byref(p))
    for k, v in overrides.items():
        setattr(p, k, v)
    return p


def certkv_live_budget(n: int, hkv: int, keep_num: int, keep_den: int) -> int:
    return int(load_library().certkv_live_budget(n, hkv, keep_num, keep_den))


def make_shape(B, L, Hq, H, n, d, w) -> certkv_shape:
    return certkv_shape(B, L, Hq, H, n, d, w)


def shape_of(K: torch.Tensor, Q_obs: Optional[torch.Tensor] = None, hq: Optional[int] = None,
             w: int = 1) -> certkv_shape:
    B, L, H, n, d = K.shape
    if Q_obs is not None:
        hq, w = Q_obs.shape[2], Q_obs.shape[3]
    return certkv_shape(B, L, hq if hq is not None else H, H, n, d, w)


def certkv_workspace_bytes(shape: certkv_shape, params: Optional[certkv_params] = None) -> int:
    params = params or certkv_default_params()
    return int(load_library().certkv_workspace_bytes(ctypes.byref(shape), ctypes.byref(params)))


def certkv_host_workspace_bytes(shape: certkv_shape, params: Optional[certkv_params] = None,
                                chunk: int = 0) -> int:
    params = params or certkv_default_params()
    return int(load_library().certkv_host_workspace_bytes(ctypes.byref(shape),
                                                          ctypes.byref(params), int(chunk)))


def certkv_decode_workspace_bytes(shape: certkv_shape) -> int:
    return int(load_library().certkv_decode_workspace_bytes(ctypes.byref(shape)))


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tensors passed to the CertKV library must be contiguous CUDA tensors")
    return ctypes.c_void_p(t.data_ptr())


def _host_ptr(t: torch.Tensor):
    if t.is_cuda or not t.is_contiguous():
        raise ValueError("host inputs must be contiguous CPU tensors (pinned for asynchronous copies)")
    return ctypes.c_void_p(t.data_ptr())


def _bf16(t: torch.Tensor, name: str) -> torch.Tensor:
    if t.dtype != torch.bfloat16:
        raise TypeError(f"{name} must be bfloat16")
    return t


def workspace(nbytes: int, device) -> torch.Tensor:
    """A caller-owned device workspace (torch allocates; the library never does)."""
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


@dataclass
class Packed:
    """Caller-owned packed cache (see certkv_packed in include/certkv.h)."""
    k: torch.Tensor
    v: torch.Tensor
    offsets: torch.Tensor
    real_counts: torch.Tensor
    positions: torch.Tensor
    tail_f32: Optional[torch.Tensor] = None
    tail_mass: Optional[torch.Tensor] = None
    tail_slot: int = 1
    clusters: int = 0
    cluster_meta: Optional[torch.Tensor] = None  # fp32 [units][m][4]
    kept_vmax: Optional[torch.Tensor] = None     # fp32 [units]

    def struct(self) -> certkv_packed:
        return certkv_packed(_ptr(self.k), _ptr(self.v), _ptr(self.offsets),
                             _ptr(self.real_counts), _ptr(self.positions), self.k.shape[0],
                             _ptr(self.tail_f32), _ptr(self.tail_mass), _ptr(self.cluster_meta),
                             _ptr(self.kept_vmax))

    def host_struct(self) -> certkv_packed:
        """The struct of a host copy (Packed.empty_host): k, v, offsets,
        real_counts, positions only."""
        return certkv_packed(_host_ptr(self.k), _host_ptr(self.v), _host_ptr(self.offsets),
                             _host_ptr(self.real_counts), _host_ptr(self.positions),
                             self.k.shape[0], None, None, None, None)

    @staticmethod
    def empty_host(B: int, L: int, H: int, d: int, B_live: int, pin: bool = True) -> "Packed":
        """Host (pinned) buffers for the packed cache copied back by
        certkv_compress_host(..., host_out=...)."""
        slots, units = B * L * B_live, B * L * H
        return Packed(k=torch.empty((slots, d), dtype=torch.bfloat16, pin_memory=pin),
                      v=torch.empty((slots, d), dtype=torch.bfloat16, pin_memory=pin),
                      offsets=torch.empty(units + 1, dtype=torch.int64, pin_memory=pin),
                      real_counts=torch.empty(units, dtype=torch.int32, pin_memory=pin),
                      positions=torch.empty(slots, dtype=torch.int32, pin_memory=pin))

    @staticmethod
    def empty(B: int, L: int, H: int, d: int, B_live: int, device, with_tail: bool = False,
              tail_slot: int = 1, clusters: int = 0) -> "Packed":
        slots = B * L * B_live
        units = B * L * H
        return Packed(
            clusters=clusters,
            cluster_meta=(torch.empty((units, clusters, 4), dtype=torch.float32, device=device)
                          if clusters else None),
            kept_vmax=(torch.empty(units, dtype=torch.float32, device=device)
                       if clusters else None),
            k=torch.empty((slots, d), dtype=torch.bfloat16, device=device),
            v=torch.empty((slots, d), dtype=torch.bfloat16, device=device),
            offsets=torch.empty(units + 1, dtype=torch.int64, device=device),
            real_counts=torch.empty(units, dtype=torch.int32, device=device),
            positions=torch.empty(slots, dtype=torch.int32, device=device),
            tail_f32=(torch.empty((units, 2, d), dtype=torch.float32, device=device)
                      if with_tail else None),
            tail_mass=(torch.empty(units, dtype=torch.float64, device=device)
                       if with_tail else None),
            tail_slot=tail_slot)


def certkv_score(K, Q_obs, params=None, *, a_out=None, ws=None, stream=None) -> torch.Tensor:
    """a1-a2: fp32 scores [B*L*H][n]."""
    _bf16(K, "K"); _bf16(Q_obs, "Q_obs")
    params = params or certkv_default_params()
    shape = shape_of(K, Q_obs)
    units = shape.batch * shape.layers * shape.hkv
    if a_out is None:
        a_out = torch.empty((units, shape.n), dtype=torch.float32, device=K.device)
    if ws is None:
        ws = workspace(certkv_workspace_bytes(shape, params), K.device)
    rc = load_library().certkv_score(ctypes.byref(shape), _ptr(K), _ptr(Q_obs),
                                     ctypes.byref(params), _ptr(a_out), _ptr(ws), ws.numel(),
                                     _stream(stream))
    _check(rc, "certkv_score")
    return a_out


def certkv_curves(V, a, params=None, *, hq: Optional[int] = None, w: int = 1, ws=None,
                  stream=None):
    """a3-a4: (perm int32 [U][n], c float64 [U][n])."""
    _bf16(V, "V")
    params = params or certkv_default_params()
    shape = shape_of(V, None, hq=hq, w=w)
    units = shape.batch * shape.layers * shape.hkv
    perm = torch.empty((units, shape.n), dtype=torch.int32, device=V.device)
    c = torch.empty((units, shape.n), dtype=torch.float64, device=V.device)
    if ws is None:
        ws = workspace(certkv_workspace_bytes(shape, params), V.device)
    rc = load_library().certkv_curves(ctypes.byref(shape), _ptr(V), _ptr(a), ctypes.byref(params),
                                      _ptr(perm), _ptr(c), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "certkv_curves")
    return perm, c


def certkv_compress_scored(K, V, a, budget_live: int, params=None, *, hq: Optional[int] = None,
                           w: int = 1, out: Optional[Packed] = None, ws=None,
                           with_tail: bool = False, stream=None) -> Packed:
    """a3-a8 from given scores."""
    _bf16(K, "K"); _bf16(V, "V")
    params = params or certkv_default_params()
    shape = shape_of(K, None, hq=hq, w=w)
    if out is None:
        out = Packed.empty(shape.batch, shape.layers, shape.hkv, shape.d, budget_live, K.device,
                           with_tail, params.tail_slot, params.tail_clusters)
    if ws is None:
        ws = workspace(certkv_workspace_bytes(shape, params), K.device)
    st = out.struct()
    rc = load_library().certkv_compress_scored(ctypes.byref(shape), _ptr(K), _ptr(V), _ptr(a),
                                               int(budget_live), ctypes.byref(params),
                                               ctypes.byref(st), _ptr(ws), ws.numel(),
                                               _stream(stream))
    _check(rc, "certkv_compress_scored")
    return out


def certkv_compress(K, V, Q_obs, budget_live: int, params=None, *, out: Optional[Packed] = None,
                    ws=None, with_tail: bool = False, stream=None) -> Packed:
    """a1-a8: the whole compression pass."""
    _bf16(K, "K"); _bf16(V, "V"); _bf16(Q_obs, "Q_obs")
    params = params or certkv_default_params()
    shape = shape_of(K, Q_obs)
    if out is None:
        out = Packed.empty(shape.batch, shape.layers, shape.hkv, shape.d, budget_live, K.device,
                           with_tail, params.tail_slot, params.tail_clusters)
    if ws is None:
        ws = workspace(certkv_workspace_bytes(shape, params), K.device)
    st = out.struct()
    rc = load_library().certkv_compress(ctypes.byref(shape), _ptr(K), _ptr(V), _ptr(Q_obs),
                                        int(budget_live), ctypes.byref(params), ctypes.byref(st),
                                        _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "certkv_compress")
    return out


def certkv_compress_host(hK, hV, hQ_obs, budget_live: int, params=None, *, chunk: int = 0,
                         out: Optional[Packed] = None, ws=None, device=None, with_tail: bool = False,
                         host_out: Optional[Packed] = None, stream=None) -> Packed:
    """a1-a8 from host tensors, copies overlapped with the compression; with
    host_out (Packed.empty_host) the packed cache is also copied back chunk by
    chunk (certkv_compress_host_copyback)."""
    _bf16(hK, "K"); _bf16(hV, "V"); _bf16(hQ_obs, "Q_obs")
    params = params or certkv_default_params()
    shape = shape_of(hK, hQ_obs)
    device = torch.device(device) if device is not None else torch.device("cuda",
                                                                          torch.cuda.current_device())
    if out is None:
        out = Packed.empty(shape.batch, shape.layers, shape.hkv, shape.d, budget_live, device,
                           with_tail, params.tail_slot, params.tail_clusters)
    if ws is None:
        ws = workspace(certkv_host_workspace_bytes(shape, params, chunk), device)
    st = out.struct()
    if host_out is not None:
        hst = host_out.host_struct()
        rc = load_library().certkv_compress_host_copyback(
            ctypes.byref(shape), _host_ptr(hK), _host_ptr(hV), _host_ptr(hQ_obs), int(budget_live),
            ctypes.byref(params), int(chunk), ctypes.byref(st), ctypes.byref(hst), _ptr(ws),
            ws.numel(), _stream(stream))
        _check(rc, "certkv_compress_host_copyback")
        return out
    rc = load_library().certkv_compress_host(ctypes.byref(shape), _host_ptr(hK), _host_ptr(hV),
                                             _host_ptr(hQ_obs),
                                             int(budget_live), ctypes.byref(params), int(chunk),
                                             ctypes.byref(st), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "certkv_compress_host")
    return out


def certkv_decode_attn(q, packed: Packed, *, hkv: int, scale: float = 0.0, out=None, ws=None,
                       stream=None) -> torch.Tensor:
    """a9: decode attention over the packed cache.  q bf16 [B][L][Hq][d]."""
    _bf16(q, "q")
    B, L, Hq, d = q.shape
    shape = certkv_shape(B, L, Hq, hkv, 2, d, 1)  # n and w are not used by decode
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        ws = workspace(certkv_decode_workspace_bytes(shape), q.device)
    st = packed.struct()
    rc = load_library().certkv_decode_attn(ctypes.byref(shape), _ptr(q), ctypes.byref(st),
                                           float(scale), int(packed.tail_slot), _ptr(out),
                                           _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "certkv_decode_attn")
    return out


def certkv_decode_certified(q, packed: Packed, *, hkv: int, scale: float = 0.0, out=None,
                            bound=None, certified=None, ws=None, stream=None):
    """Clustered-tail decode with its runtime error bound: (out bf16 [B][L][Hq][d],
    bound fp32 [B][L][Hq], certified int32 [B][L][Hq])."""
    _bf16(q, "q")
    if packed.clusters < 1:
        raise ValueError("packed cache has no cluster summaries (params.tail_clusters = 0)")
    B, L, Hq, d = q.shape
    shape = certkv_shape(B, L, Hq, hkv, 2, d, 1)
    if out is None:
        out = torch.empty_like(q)
    if bound is None:
        bound = torch.empty((B, L, Hq), dtype=torch.float32, device=q.device)
    if certified is None:
        certified = torch.empty((B, L, Hq), dtype=torch.int32, device=q.device)
    if ws is None:
        ws = workspace(certkv_decode_workspace_bytes(shape), q.device)
    st = packed.struct()
    rc = load_library().certkv_decode_certified(ctypes.byref(shape), _ptr(q), ctypes.byref(st),
                                                float(scale), int(packed.tail_slot),
                                                int(packed.clusters), _ptr(out), _ptr(bound),
                                                _ptr(certified), _ptr(ws), ws.numel(),
                                                _stream(stream))
    _check(rc, "certkv_decode_certified")
    return out, bound, certified


FIXED_ROW_FIELDS = ("kept_mass", "norm_O", "err_subset", "norm_correction", "mass_bound",
                    "err_decode", "v_max", "factorization_residual", "tail_mass", "slot_weight",
                    "l1_tail_weights", "logpartition_gap", "lift_bound", "tanh_bound",
                    "l1_lifted_row", "slot_mixture_error")


def certkv_fixed_row_stats(q, K, V, packed: Packed, *, scores=None, scale: float = 0.0,
                           stats=None, ws=None, stream=None) -> torch.Tensor:
    """Fixed-row diagnostics per query head: fp32 [B][L][Hq][16] in the order
    of FIXED_ROW_FIELDS (evaluation tool; reads the full K and V).  `scores`:
    fp32 [B*L*H][n] compression scores (certkv_score), or None (the fields
    that need the slot's tail weights are then NaN)."""
    _bf16(q, "q"); _bf16(K, "K"); _bf16(V, "V")
    B, L, Hq, d = q.shape
    shape = certkv_shape(B, L, Hq, K.shape[2], K.shape[3], d, 1)
    if scores is not None:
        if scores.dtype != torch.float32 or not scores.is_contiguous() or \
                scores.numel() != B * L * K.shape[2] * K.shape[3]:
            raise ValueError("scores must be contiguous fp32 [B*L*H][n]")
    if stats is None:
        stats = torch.empty((B, L, Hq, len(FIXED_ROW_FIELDS)), dtype=torch.float32,
                            device=q.device)
    if ws is None:
        ws = workspace(int(load_library().certkv_fixed_row_workspace_bytes(ctypes.byref(shape))),
                       q.device)
    st = packed.struct()
    rc = load_library().certkv_fixed_row_stats(ctypes.byref(shape), _ptr(q), _ptr(K), _ptr(V),
                                               _ptr(scores), ctypes.byref(st), float(scale),
                                               int(packed.tail_slot), _ptr(stats), _ptr(ws),
                                               ws.numel(), _stream(stream))
    _check(rc, "certkv_fixed_row_stats")
    return stats


def certkv_coverage_profile(q, K, *, eta=(0.1,), rel_eps=(0.1,), abs_eps=(), scale: float = 0.0,
                            with_order: bool = False, with_gap: bool = False, ws=None,
                            stream=None) -> dict:
    """Coverage profile of the decode query rows q [B][L][Hq][d] over the keys K
    [B][L][H][n][d]: K_eta int32 [B][L][Hq][len(eta)], rel / abs counts int32,
    top fp32 [B][L][Hq][2] (max logit, log-partition), and optionally order
    int32 / gap fp32 [B][L][Hq][n] (evaluation instrument; reads all of K)."""
    _bf16(q, "q"); _bf16(K, "K")
    B, L, Hq, d = q.shape
    n = K.shape[3]
    shape = certkv_shape(B, L, Hq, K.shape[2], n, d, 1)
    dev = q.device

    def host(x):
        return (ctypes.c_double * max(len(x), 1))(*[float(v) for v in x])

    def out(cnt, dtype):
        return torch.empty((B, L, Hq, cnt), dtype=dtype, device=dev) if cnt else None

    K_eta, rel, ab = out(len(eta), torch.int32), out(len(rel_eps), torch.int32), \
        out(len(abs_eps), torch.int32)
    top = torch.empty((B, L, Hq, 2), dtype=torch.float32, device=dev)
    order = out(n, torch.int32) if with_order else None
    gap = out(n, torch.float32) if with_gap else None
    if ws is None:
        ws = workspace(int(load_library().certkv_coverage_workspace_bytes(ctypes.byref(shape))),
                       dev)
    rc = load_library().certkv_coverage_profile(
        ctypes.byref(shape), _ptr(q), _ptr(K), float(scale), host(eta), len(eta), host(rel_eps),
        len(rel_eps), host(abs_eps), len(abs_eps), _ptr(K_eta), _ptr(rel), _ptr(ab), _ptr(top),
        _ptr(order), _ptr(gap), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "certkv_coverage_profile")
    return dict(K_eta=K_eta, rel=rel, abs=ab, top=top, order=order, gap=gap)


SAMPLED_FIELDS = ("kept_mass", "q_tail", "norm_correction", "err_weighted", "err_uniform",
                  "rmse_weighted", "rmse_uniform", "tail_value_variance")


def certkv_sampled_compensation(q, K, V, packed: Packed, unif, m: int, *, scale: float = 0.0,
                                stats=None, idx=None, ws=None, stream=None):
    """Sampled tail compensation per query head (evaluation tool; reads the full
    K and V): unif fp32 [B][L][Hq][2m] uniforms in [0, 1).  Returns (stats fp32
    [B][L][Hq][8] in the order of SAMPLED_FIELDS, idx int32 [B][L][Hq][2m])."""
    _bf16(q, "q"); _bf16(K, "K"); _bf16(V, "V")
    B, L, Hq, d = q.shape
    shape = certkv_shape(B, L, Hq, K.shape[2], K.shape[3], d, 1)
    if unif.dtype != torch.float32 or not unif.is_contiguous() or unif.numel() != B * L * Hq * 2 * m:
        raise ValueError("unif must be contiguous fp32 [B][L][Hq][2m]")
    if stats is None:
        stats = torch.empty((B, L, Hq, 8), dtype=torch.float32, device=q.device)
    if idx is None:
        idx = torch.empty((B, L, Hq, 2 * m), dtype=torch.int32, device=q.device)
    if ws is None:
        ws = workspace(int(load_library().certkv_sampled_workspace_bytes(ctypes.byref(shape))),
                       q.device)
    st = packed.struct()
    rc = load_library().certkv_sampled_compensation(
        ctypes.byref(shape), _ptr(q), _ptr(K), _ptr(V), ctypes.byref(st), float(scale), int(m),
        _ptr(unif), _ptr(idx), _ptr(stats), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "certkv_sampled_compensation")
    return stats, idx


def certkv_workspace_guard_arm(ws: torch.Tensor, shape: certkv_shape, params=None,
                               stream=None) -> None:
    """Fill the guard words after every region of a compression workspace."""
    params = params or certkv_default_params()
    rc = load_library().certkv_workspace_guard_arm(ctypes.byref(shape), ctypes.byref(params),
                                                   _ptr(ws), ws.numel() * ws.element_size(),
                                                   _stream(stream))
    if rc != 0:
        raise RuntimeError("certkv_workspace_guard_arm failed")


def certkv_workspace_guard_check(ws: torch.Tensor, shape: certkv_shape, params=None,
                                 stream=None) -> int:
    """Number of guard words that no longer hold their pattern (0: none)."""
    params = params or certkv_default_params()
    rc = load_library().certkv_workspace_guard_check(ctypes.byref(shape), ctypes.byref(params),
                                                     _ptr(ws), ws.numel() * ws.element_size(),
                                                     _stream(stream))
    if rc < 0:
        raise RuntimeError("certkv_workspace_guard_check failed")
    return rc


def certkv_read_status(ws: torch.Tensor, stream=None) -> int:
    """Synchronise and return the device status word left in `ws`."""
    return int(load_library().certkv_read_status(_ptr(ws), _stream(stream)))


def certkv_trace_enable(on: bool = True) -> None:
    """Bracket every library kernel launch with CUDA events (profiling aid)."""
    _check(load_library().certkv_trace_enable(1 if on else 0), "certkv_trace_enable")


def certkv_trace_report() -> dict:
    """{kernel name: (launches, total ms)} since the last report; clears it."""
    buf = ctypes.create_string_buffer(1 << 16)
    n = load_library().certkv_trace_report(buf, len(buf))
    if n < 0:
        raise RuntimeError("certkv_trace_report failed")
    out = {}
    for line in buf.value.decode().splitlines():
        name, cnt, ms = line.split()
        out[name] = (int(cnt), float(ms))
    return out


def certkv_decode_attn_noalloc(q, packed: Packed, *, hkv: int, scale: float = 0.0, out=None,
                               stream=None) -> torch.Tensor:
    """a9 for callers that cannot provide scratch memory: the library uses its
    own fixed 16 MiB device array instead (see include/certkv.h for the limit
    and for calls that overlap on the GPU).  The output tensor is the caller's."""
    _bf16(q, "q")
    B, L, Hq, d = q.shape
    shape = certkv_shape(B, L, Hq, hkv, 2, d, 1)
    if out is None:
        out = torch.empty_like(q)
    st = packed.struct()
    rc = load_library().certkv_decode_attn_noalloc(ctypes.byref(shape), _ptr(q),
                                                   ctypes.byref(st), float(scale),
                                                   int(packed.tail_slot), _ptr(out),
                                                   _stream(stream))
    _check(rc, "certkv_decode_attn_noalloc")
    return out
