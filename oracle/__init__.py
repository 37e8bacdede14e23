"""ctypes binding of the CPU oracle (kvx_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and
bench.py's cpu_baseline / reference legs.  The product library never imports
this package; the two share no code.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvx_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libkvx_oracle.so")
_lib = None

I32P = ctypes.POINTER(ctypes.c_int32)
F64P = ctypes.POINTER(ctypes.c_double)
F32P = ctypes.POINTER(ctypes.c_float)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, no fast-math)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class RopeSched(ctypes.Structure):
    _fields_ = [("base", ctypes.c_double), ("type", ctypes.c_int32), ("factor", ctypes.c_double),
                ("low", ctypes.c_double), ("high", ctypes.c_double), ("orig_ctx", ctypes.c_int32),
                ("rot", ctypes.c_int32)]


def rope_sched(g=None, base: Optional[float] = None) -> RopeSched:
    """The rotary schedule of a geometry object (attributes rope_base, rope_type, rope_factor,
    rope_low_freq_factor, rope_high_freq_factor, rope_original_max_position, rotary_dim; missing
    ones mean the plain schedule over the whole head), or the plain schedule of `base`."""
    if g is None:
        return RopeSched(float(base), 0, 1.0, 1.0, 1.0, 1, 0)
    return RopeSched(float(g.rope_base), int(getattr(g, "rope_type", 0)), float(getattr(g, "rope_factor", 1.0)),
                     float(getattr(g, "rope_low_freq_factor", 1.0)), float(getattr(g, "rope_high_freq_factor", 4.0)),
                     int(getattr(g, "rope_original_max_position", 8192)), int(getattr(g, "rotary_dim", 0)))


class Problem(ctypes.Structure):
    _fields_ = [
        ("Ls", ctypes.c_int32), ("Hs", ctypes.c_int32), ("ds", ctypes.c_int32), ("rope_s", RopeSched),
        ("Lt", ctypes.c_int32), ("Ht", ctypes.c_int32), ("dt", ctypes.c_int32), ("rope_t", RopeSched),
        ("layer_map", I32P),
        ("batch", ctypes.c_int32), ("s_max", ctypes.c_int32), ("t_max", ctypes.c_int32),
        ("src_len", I32P), ("tgt_seq_off", I32P),
        ("span_lo", I32P), ("span_hi", I32P),
        ("src_pos", I32P), ("tgt_pos", I32P),
        ("src_k", ctypes.POINTER(F32P)), ("src_v", ctypes.POINTER(F32P)),
        ("w_k", F32P), ("w_v", F32P),
        ("form", ctypes.c_int32), ("k_layers", ctypes.c_int32), ("rank", ctypes.c_int32),
        ("a_k", F32P), ("b_k", F32P), ("a_v", F32P), ("b_v", F32P),
    ]


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        _lib.kvxo_layer_map_nearest.argtypes = [ctypes.c_int, ctypes.c_int, I32P]
        _lib.kvxo_build_alignment.argtypes = [ctypes.c_int, I32P, I32P, I32P, I32P, I32P, I32P]
        _lib.kvxo_rope.argtypes = [F64P, ctypes.c_int, ctypes.c_double, ctypes.c_double, ctypes.c_int]
        _lib.kvxo_rope.restype = None
        _lib.kvxo_rope_sched_apply.argtypes = [F64P, ctypes.c_int, ctypes.POINTER(RopeSched), ctypes.c_double,
                                               ctypes.c_int]
        _lib.kvxo_rope_sched_apply.restype = None
        _lib.kvxo_rope_cache.argtypes = [F32P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                         ctypes.POINTER(RopeSched), I32P, ctypes.c_int]
        _lib.kvxo_rope_cache.restype = None
        _lib.kvxo_translate_row.argtypes = [ctypes.POINTER(Problem), ctypes.c_int, ctypes.c_int,
                                            ctypes.c_int, ctypes.c_int, F64P]
        _lib.kvxo_translate.argtypes = [ctypes.POINTER(Problem), F64P, F64P]
        _lib.kvxo_input_row.argtypes = [ctypes.POINTER(Problem), ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int, F64P]
        _lib.kvxo_group_in.argtypes = [ctypes.POINTER(Problem)]
        _lib.kvxo_fit.argtypes = [ctypes.POINTER(Problem), ctypes.POINTER(F32P), ctypes.POINTER(F32P),
                                  ctypes.c_double, F64P, F64P]
    return _lib


def _p(a, typ):
    return a.ctypes.data_as(typ) if a is not None else ctypes.cast(None, typ)


def _i32(a):
    return None if a is None else np.ascontiguousarray(a, np.int32)


def layer_map_nearest(Ls: int, Lt: int) -> np.ndarray:
    out = np.zeros(Lt, np.int32)
    if lib().kvxo_layer_map_nearest(Ls, Lt, _p(out, I32P)):
        raise ValueError("bad layer counts")
    return out


def build_alignment(src_seq_off, src_end, tgt_seq_off, tgt_end):
    src_seq_off, src_end = _i32(src_seq_off), _i32(src_end)
    tgt_seq_off, tgt_end = _i32(tgt_seq_off), _i32(tgt_end)
    T = int(tgt_seq_off[-1])
    lo = np.zeros(T, np.int32)
    hi = np.zeros(T, np.int32)
    n = lib().kvxo_build_alignment(len(tgt_seq_off) - 1, _p(src_seq_off, I32P), _p(src_end, I32P),
                                   _p(tgt_seq_off, I32P), _p(tgt_end, I32P), _p(lo, I32P), _p(hi, I32P))
    return lo, hi, n


def rope(x: np.ndarray, base: float, pos: float, sign: int) -> np.ndarray:
    """Plain-schedule rotary map of one head vector (double)."""
    v = np.array(x, np.float64).copy()
    lib().kvxo_rope(_p(v, F64P), v.shape[-1], base, float(pos), sign)
    return v


def rope_g(x: np.ndarray, geom, pos: float, sign: int) -> np.ndarray:
    """Rotary map of one head vector under geometry `geom`'s frequency schedule (double)."""
    v = np.array(x, np.float64).copy()
    r = rope_sched(geom)
    lib().kvxo_rope_sched_apply(_p(v, F64P), v.shape[-1], ctypes.byref(r), float(pos), sign)
    return v


def rope_cache(x: np.ndarray, base, pos: Optional[np.ndarray] = None, sign: int = +1) -> np.ndarray:
    """x: [B, H, S, d] float32; returns a rotated copy (float32).  `base` is a number (plain
    schedule) or a geometry object carrying its schedule."""
    y = np.ascontiguousarray(x, np.float32).copy()
    B, H, S, d = y.shape
    pos = _i32(pos)
    r = rope_sched(base=base) if isinstance(base, (int, float)) else rope_sched(base)
    lib().kvxo_rope_cache(_p(y, F32P), B, H, S, d, ctypes.byref(r), _p(pos, I32P), sign)
    return y


class OracleProblem:
    """Holds numpy arrays alive for the ctypes Problem struct."""

    def __init__(self, src_geom, dst_geom, layer_map, src_len, tgt_seq_off, s_max, t_max,
                 src_k: Sequence[np.ndarray], src_v: Sequence[np.ndarray], w_k, w_v,
                 span_lo=None, span_hi=None, src_pos=None, tgt_pos=None, form: int = 0, k_layers: int = 1,
                 low_rank=None):
        """layer_map: [Lt] or [Lt, k_layers] source layers.  form 0: GQA group, 1: dense (all
        source heads).  low_rank: (A_K, B_K, A_V, B_V) latent adapter factors; w_k/w_v are then
        ignored (pass None)."""
        self.keep = []

        def keep(a):
            self.keep.append(a)
            return a

        lm = keep(_i32(np.asarray(layer_map).reshape(-1)))
        sl = keep(_i32(src_len))
        so = keep(_i32(tgt_seq_off))
        lo, hi = keep(_i32(span_lo)), keep(_i32(span_hi))
        sp, tp = keep(_i32(src_pos)), keep(_i32(tgt_pos))
        ks = [keep(np.ascontiguousarray(a, np.float32)) for a in src_k]
        vs = [keep(np.ascontiguousarray(a, np.float32)) for a in src_v]
        kp = keep((F32P * len(ks))(*[_p(a, F32P) for a in ks]))
        vp = keep((F32P * len(vs))(*[_p(a, F32P) for a in vs]))
        f32 = lambda a: None if a is None else keep(np.ascontiguousarray(a, np.float32))
        wk, wv = f32(w_k), f32(w_v)
        ak, bk, av, bv = (None,) * 4 if low_rank is None else tuple(f32(a) for a in low_rank)
        rank = 0 if low_rank is None else int(np.asarray(low_rank[0]).shape[-1])
        self.T = int(so[-1])
        self.Lt, self.Ht, self.dt = dst_geom.num_layers, dst_geom.num_kv_heads, dst_geom.head_dim
        self.p = Problem(src_geom.num_layers, src_geom.num_kv_heads, src_geom.head_dim, rope_sched(src_geom),
                         dst_geom.num_layers, dst_geom.num_kv_heads, dst_geom.head_dim, rope_sched(dst_geom),
                         _p(lm, I32P), len(sl), s_max, t_max, _p(sl, I32P), _p(so, I32P),
                         _p(lo, I32P), _p(hi, I32P), _p(sp, I32P), _p(tp, I32P),
                         ctypes.cast(kp, ctypes.POINTER(F32P)), ctypes.cast(vp, ctypes.POINTER(F32P)),
                         _p(wk, F32P), _p(wv, F32P), int(form), int(k_layers), rank,
                         _p(ak, F32P), _p(bk, F32P), _p(av, F32P), _p(bv, F32P))

    def translate(self):
        """Returns (K, V), each [Lt, Ht, T_total, dt] float64."""
        ok = np.zeros((self.Lt, self.Ht, self.T, self.dt), np.float64)
        ov = np.zeros_like(ok)
        if lib().kvxo_translate(ctypes.byref(self.p), _p(ok, F64P), _p(ov, F64P)):
            raise ValueError("oracle: unsupported geometry")
        return ok, ov

    def input_row(self, j: int, h: int, kv: int, tp: int) -> np.ndarray:
        """The translator's input row (span mean of un-rotated source rows) of one target token."""
        out = np.zeros(lib().kvxo_group_in(ctypes.byref(self.p)), np.float64)
        if lib().kvxo_input_row(ctypes.byref(self.p), j, h, kv, tp, _p(out, F64P)):
            raise ValueError("oracle: unsupported geometry")
        return out

    def fit(self, tgt_k: Sequence[np.ndarray], tgt_v: Sequence[np.ndarray], lam: float):
        """Closed-form ridge fit of W_K, W_V against the target model's own caches
        (per target layer [B, Ht, t_max, dt] float32).  Returns two [Lt, Ht, in, dt] float64."""
        tk = [np.ascontiguousarray(a, np.float32) for a in tgt_k]
        tv = [np.ascontiguousarray(a, np.float32) for a in tgt_v]
        kp = (F32P * len(tk))(*[_p(a, F32P) for a in tk])
        vp = (F32P * len(tv))(*[_p(a, F32P) for a in tv])
        din = lib().kvxo_group_in(ctypes.byref(self.p))
        wk = np.zeros((self.Lt, self.Ht, din, self.dt), np.float64)
        wv = np.zeros_like(wk)
        rc = lib().kvxo_fit(ctypes.byref(self.p), ctypes.cast(kp, ctypes.POINTER(F32P)),
                            ctypes.cast(vp, ctypes.POINTER(F32P)), float(lam), _p(wk, F64P), _p(wv, F64P))
        if rc:
            raise ValueError(f"oracle fit failed ({rc})")
        return wk, wv

    def row(self, j: int, h: int, kv: int, tp: int) -> np.ndarray:
        out = np.zeros(self.dt, np.float64)
        if lib().kvxo_translate_row(ctypes.byref(self.p), j, h, kv, tp, _p(out, F64P)):
            raise ValueError("oracle: unsupported geometry")
        return out
