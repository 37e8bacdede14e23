"""kvx: GB300-native cross-model KV translation.

Thin ctypes binding of libkvx.so (C ABI in include/kvx.h).  Functions keep the
C names; they only marshal arguments (torch tensors -> device pointers,
Python values -> C structs).  Every step of the translation runs in the
library's CUDA kernels; there is no host fallback.  If the library has not
been built, loading it raises.

The translated operator is the paper's KV^_B(C) = T_theta(KV_A(C))
(Sections 4-5): layer alignment, token-span alignment, undo source RoPE,
per-KV-head projection with GQA regrouping, target RoPE, target cache write.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

from . import _build

KVX_OK, KVX_ERR_INVALID_ARG, KVX_ERR_UNSUPPORTED, KVX_ERR_CUDA, KVX_ERR_OOM, KVX_ERR_DEVICE_STATUS = range(6)
KVX_BF16, KVX_FP32 = 0, 1
KVX_PATH_AUTO, KVX_PATH_SIMT, KVX_PATH_TCGEN05 = 0, 1, 2
KVX_DEV_SPAN_CLAMPED = 0x01
KVX_DEV_POS_CLAMPED = 0x02
KVX_DEV_PAGE_INVALID = 0x04
KVX_DEV_SEQ_CLAMPED = 0x08
KVX_DEV_WAIT_TIMEOUT = 0x10
KVX_MAX_TARGET_LAYERS = 128

I32P = ctypes.POINTER(ctypes.c_int32)
VP = ctypes.c_void_p


KVX_ROPE_DEFAULT, KVX_ROPE_LINEAR, KVX_ROPE_LLAMA3 = 0, 1, 2


class kvx_model_geom(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("rope_base", ctypes.c_double),
                ("rope_type", ctypes.c_int32), ("rope_factor", ctypes.c_double),
                ("rope_low_freq_factor", ctypes.c_double), ("rope_high_freq_factor", ctypes.c_double),
                ("rope_original_max_position", ctypes.c_int32), ("rotary_dim", ctypes.c_int32)]


def model_geom(g) -> kvx_model_geom:
    """kvx_model_geom from any object with the same attribute names (the RoPE schedule and
    rotary_dim attributes are optional and default to the plain schedule over the whole head)."""
    return kvx_model_geom(g.num_layers, g.num_kv_heads, g.head_dim, g.rope_base,
                          int(getattr(g, "rope_type", 0)), float(getattr(g, "rope_factor", 1.0)),
                          float(getattr(g, "rope_low_freq_factor", 1.0)),
                          float(getattr(g, "rope_high_freq_factor", 4.0)),
                          int(getattr(g, "rope_original_max_position", 8192)),
                          int(getattr(g, "rotary_dim", 0)))


KVX_FORM_GROUPED, KVX_FORM_DENSE = 0, 1


class kvx_translator_desc(ctypes.Structure):
    _fields_ = [("src", kvx_model_geom), ("dst", kvx_model_geom), ("layer_map", I32P),
                ("dtype", ctypes.c_int32), ("max_position", ctypes.c_int32), ("path", ctypes.c_int32),
                ("form", ctypes.c_int32), ("layers_per_target", ctypes.c_int32)]


class kvx_src_kv(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("max_seq", ctypes.c_int32),
                ("k", ctypes.POINTER(VP)), ("v", ctypes.POINTER(VP)),
                ("stride_b", ctypes.c_int64), ("stride_h", ctypes.c_int64), ("stride_s", ctypes.c_int64),
                ("seq_len", VP), ("pos", VP)]


class kvx_tgt_tokens(ctypes.Structure):
    _fields_ = [("total_tokens", ctypes.c_int32), ("seq_off", VP), ("span_lo", VP), ("span_hi", VP),
                ("pos", VP)]


class kvx_dst_kv(ctypes.Structure):
    _fields_ = [("k", ctypes.POINTER(VP)), ("v", ctypes.POINTER(VP)), ("paged", ctypes.c_int32),
                ("max_seq", ctypes.c_int32),
                ("stride_b", ctypes.c_int64), ("stride_h", ctypes.c_int64), ("stride_t", ctypes.c_int64),
                ("page_table", VP), ("max_pages_per_seq", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("num_pages", ctypes.c_int32)]


class kvx_translator_info(ctypes.Structure):
    _fields_ = [("path", ctypes.c_int32), ("group_in", ctypes.c_int32), ("n_tile", ctypes.c_int32),
                ("smem_bytes", ctypes.c_int32), ("threads", ctypes.c_int32), ("num_sms", ctypes.c_int32),
                ("weight_bytes", ctypes.c_int64), ("table_bytes", ctypes.c_int64)]


EXPORTS = ["kvx_translator_create", "kvx_translator_create_low_rank", "kvx_translate", "kvx_fit_create",
           "kvx_fit_accumulate", "kvx_fit_solve", "kvx_fit_reset", "kvx_fit_tokens", "kvx_fit_destroy", "kvx_build_alignment", "kvx_layer_map_nearest",
           "kvx_get_device_status", "kvx_get_info", "kvx_launches_per_translate", "kvx_last_error",
           "kvx_destroy", "kvx_translate_static", "kvx_static_last_error", "kvx_span_plan_stats",
           "kvx_enable_peer", "kvx_translate_to_device", "kvx_debug_stall_next_translate"]
KVX_PEER_STORES, KVX_PEER_STAGED = 0, 1
KVX_STATIC_SCRATCH_BYTES = 8 << 20

_lib = None


class KvxError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"kvx status {status}: {msg}")
        self.status = status


def library_path() -> str:
    return _build.LIB


def build(force: bool = False) -> str:
    return _build.build(force=force)


def lib():
    """Load libkvx.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError(f"libkvx.so not built ({path}); run paper_2608_30963_gb300.build()")
        L = ctypes.CDLL(path)
        L.kvx_translator_create.argtypes = [ctypes.POINTER(kvx_translator_desc), VP, VP, ctypes.c_int32,
                                            ctypes.POINTER(VP)]
        L.kvx_translator_create_low_rank.argtypes = [ctypes.POINTER(kvx_translator_desc), ctypes.c_int32, VP, VP,
                                                     VP, VP, ctypes.c_int32, ctypes.POINTER(VP)]
        L.kvx_translate.argtypes = [VP, ctypes.POINTER(kvx_src_kv), ctypes.POINTER(kvx_tgt_tokens),
                                    ctypes.POINTER(kvx_dst_kv), VP]
        L.kvx_build_alignment.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, VP, VP, VP, VP, VP, VP,
                                          VP, VP]
        L.kvx_layer_map_nearest.argtypes = [ctypes.c_int32, ctypes.c_int32, I32P]
        L.kvx_get_device_status.argtypes = [VP, VP, ctypes.POINTER(ctypes.c_uint32), ctypes.c_int32]
        L.kvx_get_info.argtypes = [VP, ctypes.POINTER(kvx_translator_info)]
        L.kvx_launches_per_translate.argtypes = [VP]
        L.kvx_launches_per_translate.restype = ctypes.c_int32
        L.kvx_last_error.restype = ctypes.c_char_p
        L.kvx_destroy.argtypes = [VP]
        L.kvx_translate_static.argtypes = [ctypes.POINTER(kvx_translator_desc), VP, VP, ctypes.POINTER(kvx_src_kv),
                                           ctypes.POINTER(kvx_tgt_tokens), ctypes.POINTER(kvx_dst_kv),
                                           ctypes.POINTER(ctypes.c_uint32), VP]
        L.kvx_static_last_error.restype = ctypes.c_char_p
        L.kvx_fit_create.argtypes = [ctypes.POINTER(kvx_translator_desc), ctypes.c_double, ctypes.c_int32,
                                     ctypes.POINTER(VP)]
        L.kvx_fit_accumulate.argtypes = [VP, ctypes.POINTER(kvx_src_kv), ctypes.POINTER(kvx_tgt_tokens),
                                         ctypes.POINTER(kvx_dst_kv), VP]
        L.kvx_fit_solve.argtypes = [VP, VP, VP, ctypes.POINTER(ctypes.c_uint32), VP]
        L.kvx_fit_reset.argtypes = [VP, VP]
        L.kvx_fit_tokens.argtypes = [VP]
        L.kvx_fit_tokens.restype = ctypes.c_int64
        L.kvx_fit_destroy.argtypes = [VP]
        L.kvx_span_plan_stats.argtypes = [VP, VP, ctypes.POINTER(ctypes.c_int64)]
        L.kvx_enable_peer.argtypes = [ctypes.c_int32]
        L.kvx_debug_stall_next_translate.argtypes = [VP, ctypes.c_int32, ctypes.c_int32]
        L.kvx_translate_to_device.argtypes = [VP, ctypes.POINTER(kvx_src_kv), ctypes.POINTER(kvx_tgt_tokens),
                                              ctypes.POINTER(kvx_dst_kv), ctypes.c_int32, ctypes.c_int32,
                                              ctypes.POINTER(kvx_dst_kv), VP]
        for name in EXPORTS:
            if name not in ("kvx_last_error", "kvx_launches_per_translate", "kvx_static_last_error",
                            "kvx_fit_tokens"):
                getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


def kvx_last_error() -> str:
    return lib().kvx_last_error().decode()


def _check(status: int):
    if status != KVX_OK:
        raise KvxError(status, kvx_last_error())


# --------------------------------------------------------------------------- raw C calls
def kvx_layer_map_nearest(src_layers: int, dst_layers: int):
    out = (ctypes.c_int32 * dst_layers)()
    _check(lib().kvx_layer_map_nearest(src_layers, dst_layers, out))
    return list(out)


def kvx_translator_create(desc: kvx_translator_desc, w_k_ptr: int, w_v_ptr: int, weights_on_device: bool) -> int:
    h = VP()
    _check(lib().kvx_translator_create(ctypes.byref(desc), VP(w_k_ptr), VP(w_v_ptr), int(weights_on_device),
                                       ctypes.byref(h)))
    return h.value


def kvx_translator_create_low_rank(desc: kvx_translator_desc, rank: int, a_k_ptr: int, b_k_ptr: int, a_v_ptr: int,
                                   b_v_ptr: int, weights_on_device: bool) -> int:
    h = VP()
    _check(lib().kvx_translator_create_low_rank(ctypes.byref(desc), int(rank), VP(a_k_ptr), VP(b_k_ptr),
                                                VP(a_v_ptr), VP(b_v_ptr), int(weights_on_device), ctypes.byref(h)))
    return h.value


def kvx_translate(handle: int, src: kvx_src_kv, tgt: kvx_tgt_tokens, dst: kvx_dst_kv, stream: int = 0):
    _check(lib().kvx_translate(VP(handle), ctypes.byref(src), ctypes.byref(tgt), ctypes.byref(dst), VP(stream)))


def kvx_build_alignment(batch, total_src, total_tgt, src_seq_off, src_end, tgt_seq_off, tgt_end, span_lo, span_hi,
                        dev_status=0, stream: int = 0):
    _check(lib().kvx_build_alignment(batch, total_src, total_tgt, VP(src_seq_off), VP(src_end), VP(tgt_seq_off),
                                     VP(tgt_end), VP(span_lo), VP(span_hi), VP(dev_status), VP(stream)))


def kvx_translate_static(desc: kvx_translator_desc, w_k_ptr: int, w_v_ptr: int, src: kvx_src_kv,
                         tgt: kvx_tgt_tokens, dst: kvx_dst_kv, stream: int = 0, read_status: bool = False) -> int:
    """Allocation-free translation (see include/kvx.h).  Returns the device status word when
    read_status is set (the call then synchronises the stream), else 0."""
    bits = ctypes.c_uint32(0)
    st = lib().kvx_translate_static(ctypes.byref(desc), VP(w_k_ptr), VP(w_v_ptr), ctypes.byref(src),
                                    ctypes.byref(tgt), ctypes.byref(dst),
                                    ctypes.byref(bits) if read_status else None, VP(stream))
    if st not in (KVX_OK, KVX_ERR_DEVICE_STATUS):
        raise KvxError(st, lib().kvx_static_last_error().decode())
    return bits.value


def kvx_get_device_status(handle: int, stream: int = 0, clear: bool = True) -> int:
    bits = ctypes.c_uint32(0)
    st = lib().kvx_get_device_status(VP(handle), VP(stream), ctypes.byref(bits), int(clear))
    if st not in (KVX_OK, KVX_ERR_DEVICE_STATUS):
        _check(st)
    return bits.value


def kvx_get_info(handle: int) -> kvx_translator_info:
    info = kvx_translator_info()
    _check(lib().kvx_get_info(VP(handle), ctypes.byref(info)))
    return info


def kvx_launches_per_translate(handle: int) -> int:
    return lib().kvx_launches_per_translate(VP(handle))


def kvx_enable_peer(peer_device: int):
    _check(lib().kvx_enable_peer(peer_device))


def kvx_translate_to_device(handle: int, src: kvx_src_kv, tgt: kvx_tgt_tokens, dst: kvx_dst_kv, dst_device: int,
                            mode: int, staging: Optional[kvx_dst_kv] = None, stream: int = 0):
    _check(lib().kvx_translate_to_device(VP(handle), ctypes.byref(src), ctypes.byref(tgt), ctypes.byref(dst),
                                         dst_device, mode, None if staging is None else ctypes.byref(staging),
                                         VP(stream)))


def kvx_span_plan_stats(handle: int, stream: int = 0) -> dict:
    c = (ctypes.c_int64 * 4)()
    _check(lib().kvx_span_plan_stats(VP(handle), VP(stream), c))
    return {"subtiles": c[0], "staged_tokens": c[1], "global_tokens": c[2], "subtiles_with_global": c[3]}


def kvx_destroy(handle: int):
    _check(lib().kvx_destroy(VP(handle)))


# --------------------------------------------------------------------------- torch marshalling
def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def _ptr_array(tensors: Sequence) -> ctypes.Array:
    return (VP * len(tensors))(*[_ptr(t) for t in tensors])


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(getattr(stream, "cuda_stream", stream))


def _call_structs(src_k, src_v, src_seq_len, tgt_seq_off, total_tokens, dst_k, dst_v, span_lo, span_hi, src_pos,
                  tgt_pos, page_table, page_size, num_pages):
    """The three call structs of kvx_translate / kvx_fit_accumulate for torch tensors."""
    s0 = src_k[0]
    src = kvx_src_kv(s0.shape[0], s0.shape[2], _ptr_array(src_k), _ptr_array(src_v),
                     s0.stride(0), s0.stride(1), s0.stride(2), _ptr(src_seq_len), _ptr(src_pos))
    tgt = kvx_tgt_tokens(int(total_tokens), _ptr(tgt_seq_off), _ptr(span_lo), _ptr(span_hi), _ptr(tgt_pos))
    d0 = dst_k[0]
    if page_table is None:
        dst = kvx_dst_kv(_ptr_array(dst_k), _ptr_array(dst_v), 0, d0.shape[2], d0.stride(0), d0.stride(1),
                         d0.stride(2), None, 0, 0, 0)
    else:
        dst = kvx_dst_kv(_ptr_array(dst_k), _ptr_array(dst_v), 1, 0, 0, 0, 0, _ptr(page_table),
                         page_table.shape[1], page_size, num_pages or d0.shape[0])
    return src, tgt, dst


def _desc(src_geom, dst_geom, layer_map, dtype, max_position, path, form, layers_per_target, keep: list):
    lm = None
    if layer_map is not None:
        flat = [int(x) for row in layer_map for x in (row if hasattr(row, "__len__") else [row])]
        arr = (ctypes.c_int32 * len(flat))(*flat)
        keep.append(arr)
        lm = ctypes.cast(arr, I32P)
    return kvx_translator_desc(model_geom(src_geom), model_geom(dst_geom), lm, dtype, max_position, path, form,
                               layers_per_target)


class Fitter:
    """Owns one kvx_fitter: closed-form ridge fit of a linear translator's W_K, W_V from
    calibration batches (source caches and the target model's own caches of the same contexts)."""

    def __init__(self, src_geom, dst_geom, lam: float, layer_map: Optional[Sequence] = None, dtype: int = KVX_BF16,
                 form: int = KVX_FORM_GROUPED, layers_per_target: int = 1, chunk_tokens: int = 0,
                 max_position: int = 0):
        self._keep = []
        self.desc = _desc(src_geom, dst_geom, layer_map, dtype, max_position, KVX_PATH_AUTO, form, layers_per_target,
                          self._keep)
        h = VP()
        _check(lib().kvx_fit_create(ctypes.byref(self.desc), float(lam), int(chunk_tokens), ctypes.byref(h)))
        self.handle = h.value

    def accumulate(self, src_k: Sequence, src_v: Sequence, src_seq_len, tgt_seq_off, total_tokens: int,
                   tgt_k: Sequence, tgt_v: Sequence, *, span_lo=None, span_hi=None, src_pos=None, tgt_pos=None,
                   page_table=None, page_size: int = 16, num_pages: int = 0, stream=None):
        """Arguments as Translator.translate; tgt_k/tgt_v are the target model's own caches (read)."""
        src, tgt, dst = _call_structs(src_k, src_v, src_seq_len, tgt_seq_off, total_tokens, tgt_k, tgt_v, span_lo,
                                      span_hi, src_pos, tgt_pos, page_table, page_size, num_pages)
        _check(lib().kvx_fit_accumulate(VP(self.handle), ctypes.byref(src), ctypes.byref(tgt), ctypes.byref(dst),
                                        VP(_stream(stream))))

    def solve(self, w_k, w_v, stream=None) -> int:
        """Writes W_K, W_V (device tensors [L_t, H_t, in, out] of the cache dtype); returns the status word."""
        bits = ctypes.c_uint32(0)
        st = lib().kvx_fit_solve(VP(self.handle), VP(_ptr(w_k)), VP(_ptr(w_v)), ctypes.byref(bits),
                                 VP(_stream(stream)))
        if st not in (KVX_OK, KVX_ERR_DEVICE_STATUS):
            _check(st)
        return bits.value

    def reset(self, stream=None):
        _check(lib().kvx_fit_reset(VP(self.handle), VP(_stream(stream))))

    def tokens(self) -> int:
        return lib().kvx_fit_tokens(VP(self.handle))

    def close(self):
        if getattr(self, "handle", None):
            _check(lib().kvx_fit_destroy(VP(self.handle)))
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Translator:
    """Owns one kvx_translator.  Weights are torch tensors (host or device)
    [L_t, H_t, in, out] of the translator dtype; they are copied at creation.
    With low_rank=(A_K, B_K, A_V, B_V) ([L_t, H_t, in, rank] and [L_t, H_t, rank, out]),
    w_k and w_v are ignored and the translator is a latent adapter.  layer_map is
    [L_t] or, with layers_per_target = k > 1, [L_t, k] (nested or flat)."""

    def __init__(self, src_geom, dst_geom, w_k, w_v, layer_map: Optional[Sequence] = None,
                 dtype: int = KVX_BF16, max_position: int = 0, path: int = KVX_PATH_AUTO,
                 form: int = KVX_FORM_GROUPED, layers_per_target: int = 1, low_rank=None):
        lm = None
        if layer_map is not None:
            flat = [int(x) for row in layer_map for x in (row if hasattr(row, "__len__") else [row])]
            self._lm = (ctypes.c_int32 * len(flat))(*flat)
            lm = ctypes.cast(self._lm, I32P)
        self.desc = kvx_translator_desc(model_geom(src_geom), model_geom(dst_geom), lm, dtype, max_position, path,
                                        form, layers_per_target)
        if low_rank is not None:
            a_k, b_k, a_v, b_v = (t.contiguous() for t in low_rank)
            self.handle = kvx_translator_create_low_rank(self.desc, a_k.shape[-1], _ptr(a_k), _ptr(b_k), _ptr(a_v),
                                                         _ptr(b_v), a_k.is_cuda)
        else:
            w_k = w_k.contiguous()
            w_v = w_v.contiguous()
            self.handle = kvx_translator_create(self.desc, _ptr(w_k), _ptr(w_v), w_k.is_cuda)
        self.src_geom, self.dst_geom = src_geom, dst_geom

    def info(self) -> kvx_translator_info:
        return kvx_get_info(self.handle)

    def launches_per_translate(self) -> int:
        return kvx_launches_per_translate(self.handle)

    def translate(self, src_k: Sequence, src_v: Sequence, src_seq_len, tgt_seq_off, total_tokens: int,
                  dst_k: Sequence, dst_v: Sequence, *, span_lo=None, span_hi=None, src_pos=None, tgt_pos=None,
                  page_table=None, page_size: int = 16, num_pages: int = 0, stream=None):
        """src_k/src_v: per source layer [B, H_s, S_max, d_s] tensors (strided, d contiguous).
        dst_k/dst_v: per target layer, contiguous [B, H_t, T_max, d_t] (page_table None) or paged pools
        [num_pages, page_size, H_t, d_t]."""
        src, tgt, dst = _call_structs(src_k, src_v, src_seq_len, tgt_seq_off, total_tokens, dst_k, dst_v, span_lo,
                                      span_hi, src_pos, tgt_pos, page_table, page_size, num_pages)
        kvx_translate(self.handle, src, tgt, dst, _stream(stream))

    def translate_to_device(self, src_k: Sequence, src_v: Sequence, src_seq_len, tgt_seq_off, total_tokens: int,
                            dst_k: Sequence, dst_v: Sequence, dst_device: int, mode: int = KVX_PEER_STORES, *,
                            staging_k: Optional[Sequence] = None, staging_v: Optional[Sequence] = None,
                            span_lo=None, span_hi=None, src_pos=None, tgt_pos=None, page_table=None,
                            page_size: int = 16, num_pages: int = 0, stream=None):
        """As translate, with the target cache on device dst_device (kvx_translate_to_device):
        mode KVX_PEER_STORES writes it from the kernels, KVX_PEER_STAGED translates into
        staging_k / staging_v (current device, same layout) and copies them over."""
        src, tgt, dst = _call_structs(src_k, src_v, src_seq_len, tgt_seq_off, total_tokens, dst_k, dst_v, span_lo,
                                      span_hi, src_pos, tgt_pos, page_table, page_size, num_pages)
        stg = None
        if staging_k is not None:
            _, _, stg = _call_structs(src_k, src_v, src_seq_len, tgt_seq_off, total_tokens, staging_k, staging_v,
                                      span_lo, span_hi, src_pos, tgt_pos, page_table, page_size, num_pages)
        self._keep = (dst, stg)
        kvx_translate_to_device(self.handle, src, tgt, dst, dst_device, mode, stg, _stream(stream))

    def debug_stall_next_translate(self, unit: int, wait_us: int):
        """Diagnostics: the next translate times out its on-chip waits (kvx_debug_stall_next_translate)."""
        _check(lib().kvx_debug_stall_next_translate(VP(self.handle), unit, wait_us))

    def span_plan_stats(self, stream=None) -> dict:
        """Token-span plan of the last translate (span kernel only): sub-tiles, tokens staged in
        their sub-tile's window, tokens gathered from global memory."""
        return kvx_span_plan_stats(self.handle, _stream(stream))

    def device_status(self, stream=None, clear: bool = True) -> int:
        return kvx_get_device_status(self.handle, _stream(stream), clear)

    def close(self):
        if getattr(self, "handle", None):
            kvx_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def build_alignment(src_seq_off, src_end, tgt_seq_off, tgt_end, span_lo, span_hi, dev_status=None, stream=None):
    """Device int32 tensors in, span_lo/span_hi (device int32[T_total]) written."""
    batch = tgt_seq_off.shape[0] - 1
    kvx_build_alignment(batch, src_end.shape[0], tgt_end.shape[0], _ptr(src_seq_off), _ptr(src_end),
                        _ptr(tgt_seq_off), _ptr(tgt_end), _ptr(span_lo), _ptr(span_hi), _ptr(dev_status),
                        _stream(stream))
