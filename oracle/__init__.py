"""Float64 CPU oracle of the CertKV compression pass — TEST INFRASTRUCTURE ONLY.

This package wraps ``certkv_oracle.c`` (plain C, float64, naive loops written
from the paper's §4, Eq. (certkv-curve), Algorithm 1 and the appendix "CertKV:
implementation and exact-budget protocol").  Only the tests, the smoke check
and the benchmark's CPU-baseline leg may import it.  It shares no code with the
CUDA library and never imports it.

All arrays are numpy; bf16 tensors are passed as their raw ``uint16`` bit
patterns, widened exactly to float64 inside the C code.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "certkv_oracle.c")
_LIB_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_LIB_DIR, "liboracle_certkv.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-std=c99",
          "-D_DEFAULT_SOURCE"]


def build(force: bool = False) -> str:
    """Compile the oracle shared library (gcc) and return its path."""
    os.makedirs(_LIB_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["cc", *CFLAGS, "-o", tmp, _SRC, "-lm", "-lpthread"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _bind(lib):
    P = ctypes.c_void_p
    I, D, I64 = ctypes.c_int, ctypes.c_double, ctypes.c_int64
    lib.oracle_scores.argtypes = [P, P, I, I, I, I, D, I, I, P]
    lib.oracle_scores.restype = I
    lib.oracle_order.argtypes = [P, I, P]
    lib.oracle_order.restype = None
    lib.oracle_curve.argtypes = [P, P, P, I, I, I, P]
    lib.oracle_curve.restype = None
    lib.oracle_b_min.argtypes = [I64, I, I64, I64]
    lib.oracle_b_min.restype = I64
    lib.oracle_allocate.argtypes = [P, I, I, I64, I64, I64, I, P, P]
    lib.oracle_allocate.restype = I
    lib.oracle_allocate_mode.argtypes = [P, I, I, I64, I64, I64, I, I, P, P]
    lib.oracle_allocate_mode.restype = I
    lib.oracle_select.argtypes = [P, I, P]
    lib.oracle_select.restype = None
    lib.oracle_tail.argtypes = [P, P, P, P, I, I, I, P, P, P]
    lib.oracle_tail.restype = D
    lib.oracle_compress.argtypes = [P, D, I64, P, P, P, P, I] + [P] * 13
    lib.oracle_tail_clusters.argtypes = [P, P, P, I, I, I, I, P, P, P, P, P, P]
    lib.oracle_tail_clusters.restype = None
    lib.oracle_decode_certified.argtypes = [P, P, P, I, I, D, P, P, P, P, P, I, P, P, P]
    lib.oracle_decode_certified.restype = D
    lib.oracle_fixed_row.argtypes = [P, P, P, P, I, I, D, P, P]
    lib.oracle_fixed_row.restype = None
    lib.oracle_future_query_lift.argtypes = [P, P, P, P, P, P, P, I, I, D, P]
    lib.oracle_future_query_lift.restype = None
    lib.oracle_coverage_profile.argtypes = [P, P, I, I, D, P, I, P, I, P, I, P, P, P, P, P, P]
    lib.oracle_coverage_profile.restype = None
    lib.oracle_sampled_compensation.argtypes = [P, P, P, P, I, I, D, I, P, P, P, P]
    lib.oracle_sampled_compensation.restype = None
    lib.oracle_compress.restype = I
    lib.oracle_decode.argtypes = [P, D, P, P, P, P, P, I, P]
    lib.oracle_decode.restype = None
    lib.oracle_f64_to_bf16.argtypes = [D]
    lib.oracle_f64_to_bf16.restype = ctypes.c_uint16
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
    return _lib


def compile_variant(src_text: str, out_dir: str) -> str:
    """Compile a modified copy of the oracle source (used by the tests that
    plant a mistake in the oracle and check that a pin catches it)."""
    src = os.path.join(out_dir, "variant.c")
    lib = os.path.join(out_dir, "libvariant.so")
    with open(src, "w") as f:
        f.write(src_text)
    subprocess.run(["cc", *CFLAGS, "-o", lib, src, "-lm", "-lpthread"], check=True)
    return lib


def load_variant(path: str):
    """Bind a compiled oracle variant; pass the result as ``lib=`` to any call."""
    return _bind(ctypes.CDLL(path))


def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


def _ptr(x: np.ndarray) -> ctypes.c_void_p:
    assert x.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return ctypes.c_void_p(x.ctypes.data)


def _u16(x) -> np.ndarray:
    x = np.ascontiguousarray(x)
    if x.dtype != np.uint16:
        raise TypeError("bf16 tensors are passed as their uint16 bit patterns")
    return x


def bf16_bits_to_f64(x: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    return (np.asarray(x, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x: float, *, lib=None) -> int:
    """Round-to-nearest-even of a float64 to bf16, as the oracle packs the tail slot."""
    return int((lib or _load()).oracle_f64_to_bf16(float(x)))


# ---------------------------------------------------------------- per step --

def scores(K, Qg, w: int, G: int, scale: float, pool: int = 5, protect: int = 1, *, lib=None) -> np.ndarray:
    """a1-a2 for one unit: K [n][d] uint16, Qg [G][w][d] uint16 -> a [n] float64."""
    K = _u16(K); Qg = _u16(Qg)
    n, d = K.shape
    assert Qg.shape == (G, w, d)
    a = np.empty(n, dtype=np.float64)
    rc = (lib or _load()).oracle_scores(_ptr(K), _ptr(Qg), n, d, w, G, float(scale), int(pool),
                               int(protect), _ptr(a))
    assert rc == 0
    return a


def order(a, *, lib=None) -> np.ndarray:
    """a3: perm[r] = token at rank r (descending score, ties by lower index)."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    perm = np.empty(a.shape[0], dtype=np.int32)
    (lib or _load()).oracle_order(_ptr(a), a.shape[0], _ptr(perm))
    return perm


def curve(a, V, perm, statistic: int = 0, *, lib=None) -> np.ndarray:
    """a4: c(b) for b = 0..n-1 over the evicted ranks b..n-1."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    V = _u16(V)
    perm = np.ascontiguousarray(perm, dtype=np.int32)
    n, d = V.shape
    c = np.empty(n, dtype=np.float64)
    (lib or _load()).oracle_curve(_ptr(a), _ptr(V), _ptr(perm), n, d, int(statistic), _ptr(c))
    return c


def b_min(B_real: int, H: int, alpha_num: int = 1, alpha_den: int = 5, *, lib=None) -> int:
    return int((lib or _load()).oracle_b_min(int(B_real), int(H), int(alpha_num), int(alpha_den)))


def allocate(curves, B_real: int, alpha_num: int = 1, alpha_den: int = 5, T: int = 40, *,
             mode: int = 0, lib=None):
    """a5: per-head real-token budgets.  curves [H][n] float64.  mode 0: Lagrangian
    bisection + repair (the method); 1: true uniform; 2: greedy marginal from b_min.

    Returns (b [H] int32, repairs) or raises ValueError on an infeasible budget."""
    curves = np.ascontiguousarray(curves, dtype=np.float64)
    H, n = curves.shape
    ptrs = (ctypes.c_void_p * H)(*[curves.ctypes.data + h * n * 8 for h in range(H)])
    b = np.empty(H, dtype=np.int32)
    rep = np.zeros(1, dtype=np.int64)
    rc = (lib or _load()).oracle_allocate_mode(ctypes.cast(ptrs, ctypes.c_void_p), H, n,
                                               int(B_real), int(alpha_num), int(alpha_den),
                                               int(T), int(mode), _ptr(b), _ptr(rep))
    if rc != 0:
        raise ValueError("infeasible budget")
    return b, int(rep[0])


def select(perm, b: int, *, lib=None) -> np.ndarray:
    """a6: kept token positions (ascending) = ranks 0..b-1."""
    perm = np.ascontiguousarray(perm, dtype=np.int32)
    kept = np.empty(max(int(b), 0), dtype=np.int32)
    (lib or _load()).oracle_select(_ptr(perm), int(b), _ptr(kept))
    return kept


def tail(a, K, V, perm, b: int, *, lib=None):
    """a7: (k*, v*, m, zero_mass) over the evicted ranks b..n-1."""
    a = np.ascontiguousarray(a, dtype=np.float64)
    K = _u16(K); V = _u16(V)
    perm = np.ascontiguousarray(perm, dtype=np.int32)
    n, d = K.shape
    ks = np.empty(d, dtype=np.float64)
    vs = np.empty(d, dtype=np.float64)
    zero = np.zeros(1, dtype=np.int32)
    m = (lib or _load()).oracle_tail(_ptr(a), _ptr(K), _ptr(V), _ptr(perm), n, d, int(b), _ptr(ks),
                            _ptr(vs), _ptr(zero))
    return ks, vs, float(m), bool(zero[0])


# -------------------------------------------------------------- whole pass --

def compress(K, V, Q, *, B: int, L: int, Hq: int, H: int, n: int, d: int, w: int,
             B_live: int, scale: float = 0.0, pool: int = 5, protect: int = 1,
             alpha_num: int = 1, alpha_den: int = 5, T: int = 40, statistic: int = 0,
             tail_slot: int = 1, allocator: int = 0, clusters: int = 0, a_in=None,
             threads: int | None = None, lib=None) -> dict:
    """The whole compression pass in the packed layout of the CUDA library.

    K, V: uint16 [B][L][H][n][d]; Q: uint16 [B][L][Hq][w][d] (may be None when
    a_in, fp32 [B*L*H][n], is given: conditioned mode starting from those scores).
    """
    units = B * L * H
    K = _u16(K).reshape(units, n, d)
    V = _u16(V).reshape(units, n, d)
    if a_in is None:
        Q = _u16(Q).reshape(B * L * Hq, w, d)
    else:
        a_in = np.ascontiguousarray(a_in, dtype=np.float32).reshape(units, n)
        Q = np.zeros(1, dtype=np.uint16)
    if scale == 0.0:
        scale = 1.0 / np.sqrt(d)
    cfg = np.array([B, L, Hq, H, n, d, w, pool, protect, alpha_num, alpha_den, T,
                    statistic, tail_slot, allocator, clusters], dtype=np.int32)
    slots = B * L * B_live
    out = dict(
        a=np.empty((units, n), np.float64), perm=np.empty((units, n), np.int32),
        c=np.empty((units, n), np.float64), counts=np.empty(units, np.int32),
        offsets=np.empty(units + 1, np.int64), positions=np.empty(slots, np.int32),
        pk=np.empty((slots, d), np.uint16), pv=np.empty((slots, d), np.uint16),
        tail=np.zeros((units, 2, d), np.float64), tail_mass=np.zeros(units, np.float64),
        repairs=np.zeros(B * L, np.int64),
        cl_meta=np.zeros((units, max(clusters, 1), 3), np.float64),
        kept_vmax=np.zeros(units, np.float64))
    if threads is None:
        threads = os.cpu_count() or 1
    rc = (lib or _load()).oracle_compress(
        _ptr(cfg), float(scale), int(B_live), _ptr(K), _ptr(V), _ptr(Q),
        _ptr(a_in) if a_in is not None else None, int(threads),
        _ptr(out["a"]), _ptr(out["perm"]), _ptr(out["c"]), _ptr(out["counts"]),
        _ptr(out["offsets"]), _ptr(out["positions"]), _ptr(out["pk"]), _ptr(out["pv"]),
        _ptr(out["tail"]), _ptr(out["tail_mass"]), _ptr(out["repairs"]),
        _ptr(out["cl_meta"]), _ptr(out["kept_vmax"]))
    if rc == 2:
        raise ValueError("infeasible budget")
    out["zero_tail"] = bool(rc & 0x100)
    out["threads"] = threads
    return out


def tail_clusters(K, V, perm, b: int, m: int, *, lib=None):
    """Cluster summaries of the evicted ranks b..n-1 of one unit.  K, V uint16
    [n][d]; perm int32 [n].  Returns (kbar bits [m][d], vbar bits [m][d],
    count [m], key radius [m], value radius [m], kept value-norm max)."""
    K = _u16(K); V = _u16(V)
    n, d = K.shape
    perm = np.ascontiguousarray(perm, dtype=np.int32)
    kb = np.zeros((m, d), np.uint16); vb = np.zeros((m, d), np.uint16)
    cnt = np.zeros(m, np.int32); rk = np.zeros(m); rv = np.zeros(m); vm = np.zeros(1)
    (lib or _load()).oracle_tail_clusters(_ptr(K), _ptr(V), _ptr(perm), n, d, int(b), int(m),
                                          _ptr(kb), _ptr(vb), _ptr(cnt), _ptr(rk), _ptr(rv),
                                          _ptr(vm))
    return kb, vb, cnt, rk, rv, float(vm[0])


def decode_certified(q, pk, pv, kbar, vbar, count, rk, rv, *, scale: float, lib=None):
    """Certified decode of one query head: q uint16 [d]; kept rows pk, pv uint16
    [b][d]; clusters as from tail_clusters.  Returns (O-hat [d], bound,
    certified, structural form)."""
    q = _u16(q); pk = _u16(pk); pv = _u16(pv); kbar = _u16(kbar); vbar = _u16(vbar)
    b, d = pk.shape if pk.size else (0, q.shape[0])
    m = kbar.shape[0]
    count = np.ascontiguousarray(count, dtype=np.int32)
    rk = np.ascontiguousarray(rk, dtype=np.float64); rv = np.ascontiguousarray(rv, dtype=np.float64)
    out = np.zeros(d); cert = np.zeros(1, np.int32); struct = np.zeros(1)
    bound = (lib or _load()).oracle_decode_certified(
        _ptr(q), _ptr(pk), _ptr(pv), int(b), int(d), float(scale), _ptr(kbar), _ptr(vbar),
        _ptr(count), _ptr(rk), _ptr(rv), int(m), _ptr(out), _ptr(cert), _ptr(struct))
    return out, float(bound), bool(cert[0]), float(struct[0])


def fixed_row(q, K, V, kept, *, scale: float, ohat=None, lib=None) -> np.ndarray:
    """Fixed-row quantities of one query row over all n tokens of a unit:
    q uint16 [d], K, V uint16 [n][d], kept bool [n], ohat float64 [d] or None.
    Returns stats [8] (see oracle_fixed_row)."""
    q = _u16(q); K = _u16(K); V = _u16(V)
    n, d = K.shape
    kept = np.ascontiguousarray(kept, dtype=np.uint8)
    st = np.zeros(8)
    oh = None if ohat is None else np.ascontiguousarray(ohat, dtype=np.float64)
    (lib or _load()).oracle_fixed_row(_ptr(q), _ptr(K), _ptr(V), _ptr(kept), n, d, float(scale),
                                      _ptr(oh) if oh is not None else None, _ptr(st))
    return st


def future_query_lift(q, K, V, kept, s, *, scale: float, kstar=None, vstar=None,
                      lib=None) -> np.ndarray:
    """Future-query lift quantities of one query row (see
    oracle_future_query_lift): q uint16 [d], K, V uint16 [n][d], kept bool
    [n], s float32 [n] (the compression scores; only the tail entries are
    read), kstar, vstar uint16 [d] or None (no synthetic slot).  Returns [8]."""
    q = _u16(q); K = _u16(K); V = _u16(V)
    n, d = K.shape
    kept = np.ascontiguousarray(kept, dtype=np.uint8)
    s = np.ascontiguousarray(s, dtype=np.float32)
    ks = None if kstar is None else _u16(kstar)
    vs = None if vstar is None else _u16(vstar)
    st = np.zeros(8)
    (lib or _load()).oracle_future_query_lift(
        _ptr(q), _ptr(K), _ptr(V), _ptr(kept), _ptr(s), _ptr(ks) if ks is not None else None,
        _ptr(vs) if vs is not None else None, n, d, float(scale), _ptr(st))
    return st


def coverage_profile(q, K, *, scale: float, eta=(0.1,), rel_eps=(0.1,), abs_eps=(),
                     lib=None) -> dict:
    """Coverage profile of one query row over the n keys K (see
    oracle_coverage_profile): q uint16 [d], K uint16 [n][d].  Returns order
    int32 [n], gap float64 [n] (G(j) for ranks j = 1..n), K_eta, rel, abs
    int32 per threshold, and top = (z_(1), log sum e^z)."""
    q = _u16(q); K = _u16(K)
    n, d = K.shape
    eta = np.ascontiguousarray(eta, dtype=np.float64)
    rel_eps = np.ascontiguousarray(rel_eps, dtype=np.float64)
    abs_eps = np.ascontiguousarray(abs_eps, dtype=np.float64)
    order = np.zeros(n, np.int32)
    gap = np.zeros(n)
    K_eta = np.zeros(max(len(eta), 1), np.int32)
    rel = np.zeros(max(len(rel_eps), 1), np.int32)
    ab = np.zeros(max(len(abs_eps), 1), np.int32)
    top = np.zeros(2)
    (lib or _load()).oracle_coverage_profile(
        _ptr(q), _ptr(K), n, d, float(scale), _ptr(eta), len(eta), _ptr(rel_eps), len(rel_eps),
        _ptr(abs_eps), len(abs_eps), _ptr(order), _ptr(gap), _ptr(K_eta), _ptr(rel), _ptr(ab),
        _ptr(top))
    return dict(order=order, gap=gap, K_eta=K_eta[:len(eta)], rel=rel[:len(rel_eps)],
                abs=ab[:len(abs_eps)], top=top)


def sampled_compensation(q, K, V, kept, u, *, scale: float, m: int, forced_idx=None,
                         lib=None):
    """Sampled tail compensation of one query row (see
    oracle_sampled_compensation): q uint16 [d], K, V uint16 [n][d], kept bool
    [n], u float32 [2m] uniforms in [0, 1), forced_idx int32 [2m] or None.
    Returns (idx int32 [2m], stats [8])."""
    q = _u16(q); K = _u16(K); V = _u16(V)
    n, d = K.shape
    kept = np.ascontiguousarray(kept, dtype=np.uint8)
    if (~kept.astype(bool)).sum() < m:
        raise ValueError("m exceeds the tail")
    u = np.ascontiguousarray(u, dtype=np.float32)
    assert u.shape == (2 * m,)
    f = None if forced_idx is None else np.ascontiguousarray(forced_idx, dtype=np.int32)
    idx = np.zeros(2 * m, np.int32)
    st = np.zeros(8)
    (lib or _load()).oracle_sampled_compensation(
        _ptr(q), _ptr(K), _ptr(V), _ptr(kept), n, d, float(scale), int(m), _ptr(u),
        _ptr(f) if f is not None else None, _ptr(idx), _ptr(st))
    return idx, st


def decode(q, pk, pv, offsets, counts, *, B: int, L: int, Hq: int, H: int, d: int,
           scale: float = 0.0, tail_slot: int = 1, lib=None) -> np.ndarray:
    """a9: float64 decode attention over a packed cache.  q uint16 [B][L][Hq][d]."""
    q = _u16(q).reshape(B * L * Hq, d)
    pk = _u16(pk); pv = _u16(pv)
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    counts = np.ascontiguousarray(counts, dtype=np.int32)
    if scale == 0.0:
        scale = 1.0 / np.sqrt(d)
    cfg = np.array([B, L, Hq, H, 0, d, 0], dtype=np.int32)
    out = np.empty((B * L * Hq, d), np.float64)
    (lib or _load()).oracle_decode(_ptr(cfg), float(scale), _ptr(q), _ptr(pk), _ptr(pv),
                          _ptr(offsets), _ptr(counts), int(tail_slot), _ptr(out))
    return out.reshape(B, L, Hq, d)
