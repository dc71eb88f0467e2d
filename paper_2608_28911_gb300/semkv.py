"""Python binding of the SemKV C ABI (include/semkv.h).

Argument marshalling only: every function below forwards to the function of the
same name in libsemkv.so, passing device pointers of torch tensors and the
current CUDA stream.  PyTorch provides device memory and streams; every step of
the cache's hot path runs in the library's CUDA kernels.  If the library has not
been built (``paper_2608_28911_gb300.build.build()``) importing this module
raises: there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

import torch

from . import build as _build

BASE_AFFINE, BASE_TQ, BASE_AFFINE_HAD, BASE_TQ_DENSE = 0, 1, 2, 3
HEAD_DIM = 128

_STATUS = {0: "ok", 1: "invalid argument", 2: "misaligned pointer or capacity",
           3: "capacity exceeded", 4: "unsupported", 5: "CUDA error", 6: "workspace too small"}


class SemkvError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} failed: {_STATUS.get(status, status)} (status {status})")
        self.status = status


class QuantDescStruct(ctypes.Structure):
    _fields_ = [("base", ctypes.c_int32), ("levels_hi", ctypes.c_int32),
                ("levels_lo", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("signs", ctypes.c_void_p), ("centroids_hi", ctypes.c_void_p),
                ("thresholds_hi", ctypes.c_void_p), ("centroids_lo", ctypes.c_void_p),
                ("thresholds_lo", ctypes.c_void_p), ("rotation", ctypes.c_void_p)]


class CacheStruct(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("layers", ctypes.c_int32),
                ("kv_heads", ctypes.c_int32), ("q_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("block", ctypes.c_int32),
                ("hi_pool", ctypes.c_void_p), ("lo_pool", ctypes.c_void_p),
                ("hi_cap", ctypes.c_int64), ("lo_cap", ctypes.c_int64),
                ("hi_tok", ctypes.c_void_p), ("lo_tok", ctypes.c_void_p),
                ("hi_count", ctypes.c_int64), ("lo_count", ctypes.c_int64),
                ("n_tokens", ctypes.c_int64),
                ("stage_k", ctypes.c_void_p), ("stage_v", ctypes.c_void_p),
                ("stage_score", ctypes.c_void_p), ("stage_n", ctypes.c_int32),
                ("blk_is_high", ctypes.c_void_p), ("blk_slot", ctypes.c_void_p),
                ("dev_error", ctypes.c_void_p)]


def _load():
    path = _build.LIB
    if not os.path.exists(path):
        raise ImportError(f"libsemkv.so is not built ({path}); run "
                          "paper_2608_28911_gb300.build.build() first")
    L = ctypes.CDLL(path)
    p, i32, i64, u32, sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                            ctypes.c_size_t)
    L.semkv_row_bytes.argtypes = [i32]
    L.semkv_row_bytes.restype = sz
    L.semkv_record_bytes.argtypes = [i32, i32]
    L.semkv_record_bytes.restype = sz
    L.semkv_high_count_floor.argtypes = [u32, u32, u32]
    L.semkv_high_count_floor.restype = u32
    L.semkv_block_high_count.argtypes = [u32, u32, u32]
    L.semkv_block_high_count.restype = u32
    L.semkv_lloyd_max_gaussian.argtypes = [i32, p, p]
    L.semkv_lloyd_max_gaussian.restype = ctypes.c_int
    L.semkv_rank_workspace_bytes.argtypes = [i32, i32, i32]
    L.semkv_rank_workspace_bytes.restype = sz
    L.semkv_rank_assign.argtypes = [p, i32, i32, u32, p, p, p, p, sz, p]
    L.semkv_rank_assign.restype = ctypes.c_int
    L.semkv_score_kv_norm.argtypes = [p, i32, i32, i32, i32, i32, i32, p, p]
    L.semkv_fake_quant.argtypes = [p, p, p, i32, i32, i32, i32, p, p, p, p]
    L.semkv_fake_quant.restype = ctypes.c_int
    L.semkv_score_kv_norm.restype = ctypes.c_int
    L.semkv_quantize_pack.argtypes = [ctypes.POINTER(QuantDescStruct), p, p, i32, p, p, u32,
                                      ctypes.POINTER(CacheStruct), p]
    L.semkv_quantize_pack.restype = ctypes.c_int
    L.semkv_append_block.argtypes = [ctypes.POINTER(QuantDescStruct),
                                     ctypes.POINTER(CacheStruct), u32, u32, p]
    L.semkv_append_block.restype = ctypes.c_int
    L.semkv_decode_workspace_bytes.argtypes = [ctypes.POINTER(CacheStruct)]
    L.semkv_decode_workspace_bytes.restype = sz
    L.semkv_decode_attention.argtypes = [ctypes.POINTER(QuantDescStruct),
                                         ctypes.POINTER(CacheStruct), i32, p, p,
                                         ctypes.c_float, p, sz, p]
    L.semkv_decode_attention.restype = ctypes.c_int
    L.semkv_decode_attention_noalloc.argtypes = [ctypes.POINTER(QuantDescStruct),
                                                 ctypes.POINTER(CacheStruct), i32, p, p,
                                                 ctypes.c_float, p]
    L.semkv_decode_attention_noalloc.restype = ctypes.c_int
    L.semkv_debug_wait_timeout.argtypes = [p, u32, p]
    L.semkv_debug_wait_timeout.restype = ctypes.c_int
    L.semkv_status_string.argtypes = [ctypes.c_int]
    L.semkv_status_string.restype = ctypes.c_char_p
    return L


LIB = _load()
EXPORTED = ["semkv_row_bytes", "semkv_record_bytes", "semkv_high_count_floor",
            "semkv_block_high_count", "semkv_lloyd_max_gaussian", "semkv_rank_workspace_bytes",
            "semkv_rank_assign", "semkv_score_kv_norm", "semkv_fake_quant", "semkv_quantize_pack", "semkv_append_block",
            "semkv_decode_workspace_bytes", "semkv_decode_attention",
            "semkv_decode_attention_noalloc", "semkv_debug_wait_timeout", "semkv_status_string"]


def _ptr(t):
    if t is None:
        return None
    assert t.is_contiguous(), "tensors passed to libsemkv must be contiguous"
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(fn, status):
    if status != 0:
        raise SemkvError(fn, status)


# ------------------------------------------------------------- plain calls ----

def semkv_row_bytes(levels: int) -> int:
    return LIB.semkv_row_bytes(levels)


def semkv_record_bytes(base: int, levels: int) -> int:
    return LIB.semkv_record_bytes(base, levels)


def semkv_high_count_floor(T: int, r_num: int, r_den: int) -> int:
    return LIB.semkv_high_count_floor(T, r_num, r_den)


def semkv_block_high_count(n: int, r_num: int, r_den: int) -> int:
    return LIB.semkv_block_high_count(n, r_num, r_den)


def semkv_lloyd_max_gaussian(levels: int):
    """Host fp64 Lloyd-Max codebook -> (centroids f32 [L], thresholds f32 [L-1])."""
    c = (ctypes.c_float * levels)()
    t = (ctypes.c_float * max(levels - 1, 1))()
    _check("semkv_lloyd_max_gaussian", LIB.semkv_lloyd_max_gaussian(levels, c, t))
    return (torch.tensor(list(c), dtype=torch.float32),
            torch.tensor(list(t)[:levels - 1], dtype=torch.float32))


def semkv_rank_workspace_bytes(batch: int, T: int, want_rank: bool = True) -> int:
    return LIB.semkv_rank_workspace_bytes(batch, T, 1 if want_rank else 0)


def semkv_rank_assign(scores: torch.Tensor, n_high: int, is_high: torch.Tensor,
                      slot: torch.Tensor, rank=None, ws=None, stream=None):
    B, T = scores.shape
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size()
    _check("semkv_rank_assign",
           LIB.semkv_rank_assign(_ptr(scores), B, T, n_high, _ptr(is_high), _ptr(slot),
                                 _ptr(rank), _ptr(ws), ws_bytes, _stream(stream)))


def semkv_fake_quant(desc: "QuantDesc", k: torch.Tensor, v: torch.Tensor, k_out: torch.Tensor,
                     v_out: torch.Tensor, is_high=None, stream=None):
    """Quantize + reconstruct every row of k, v [B][NL][H][T][128] fp16 into k_out, v_out."""
    B, NL, H, T, _ = k.shape
    _check("semkv_fake_quant",
           LIB.semkv_fake_quant(ctypes.byref(desc.s), _ptr(k), _ptr(v), B, NL, H, T,
                                _ptr(is_high), _ptr(k_out), _ptr(v_out), _stream(stream)))


def semkv_score_kv_norm(x: torch.Tensor, scores: torch.Tensor, layer_begin: int = 0,
                        layer_end=None, stream=None):
    """KV-norm importance scores of x [B][NL][H][T][128] fp16 into scores [B][T] f32."""
    B, NL, H, T, _ = x.shape
    le = NL if layer_end is None else layer_end
    _check("semkv_score_kv_norm",
           LIB.semkv_score_kv_norm(_ptr(x), B, NL, H, T, layer_begin, le, _ptr(scores),
                                   _stream(stream)))


def semkv_quantize_pack(desc: "QuantDesc", k: torch.Tensor, v: torch.Tensor, is_high, slot,
                        n_high: int, cache: "KVCache", stream=None):
    T = k.shape[3]
    _check("semkv_quantize_pack",
           LIB.semkv_quantize_pack(ctypes.byref(desc.s), _ptr(k), _ptr(v), T, _ptr(is_high),
                                   _ptr(slot), n_high, ctypes.byref(cache.s), _stream(stream)))


def semkv_append_block(desc: "QuantDesc", cache: "KVCache", r_num: int, r_den: int,
                       stream=None):
    _check("semkv_append_block",
           LIB.semkv_append_block(ctypes.byref(desc.s), ctypes.byref(cache.s), r_num, r_den,
                                  _stream(stream)))


def semkv_decode_workspace_bytes(cache: "KVCache") -> int:
    return LIB.semkv_decode_workspace_bytes(ctypes.byref(cache.s))


def semkv_decode_attention(desc: "QuantDesc", cache: "KVCache", layer: int, q: torch.Tensor,
                           out: torch.Tensor, softmax_scale: float, ws: torch.Tensor,
                           stream=None):
    _check("semkv_decode_attention",
           LIB.semkv_decode_attention(ctypes.byref(desc.s), ctypes.byref(cache.s), layer,
                                      _ptr(q), _ptr(out), softmax_scale, _ptr(ws),
                                      ws.numel() * ws.element_size(), _stream(stream)))


def semkv_decode_attention_noalloc(desc: "QuantDesc", cache: "KVCache", layer: int,
                                   q: torch.Tensor, out: torch.Tensor, softmax_scale: float,
                                   stream=None):
    """Decode attention with the library's static split-K scratch (no workspace):
    for callers that cannot allocate device memory.  See include/semkv.h."""
    _check("semkv_decode_attention_noalloc",
           LIB.semkv_decode_attention_noalloc(ctypes.byref(desc.s), ctypes.byref(cache.s), layer,
                                              _ptr(q), _ptr(out), softmax_scale,
                                              _stream(stream)))


def semkv_debug_wait_timeout(dev_error: torch.Tensor, polls: int, stream=None):
    """Run the kernels' bounded mbarrier wait on a barrier nothing arrives on, giving up
    after `polls` polls: the wait reports a timeout (1) in dev_error (device int32)."""
    _check("semkv_debug_wait_timeout",
           LIB.semkv_debug_wait_timeout(_ptr(dev_error), polls, _stream(stream)))


# ------------------------------------------------------- owning wrappers ------

class QuantDesc:
    """A semkv_quant_desc whose device tables are torch tensors kept alive here."""

    def __init__(self, base: int, levels_hi: int, levels_lo: int, signs=None,
                 device="cuda", rotation=None):
        self.base, self.levels_hi, self.levels_lo = base, levels_hi, levels_lo
        self._keep = []
        s = QuantDescStruct(base=base, levels_hi=levels_hi, levels_lo=levels_lo,
                            head_dim=HEAD_DIM)
        if base in (BASE_TQ, BASE_TQ_DENSE):
            if base == BASE_TQ:
                assert signs is not None, "the TQ base needs a sign vector per (layer, head)"
                sg = torch.as_tensor(signs, dtype=torch.int8).to(device).contiguous()
                self._keep.append(sg)
                s.signs = sg.data_ptr()
                self.signs = sg
            else:
                assert rotation is not None, "the dense TQ base needs a rotation per (layer, head)"
                rt = torch.as_tensor(np.ascontiguousarray(rotation).view(np.int16)).to(device)
                self._keep.append(rt.contiguous())
                s.rotation = self._keep[-1].data_ptr()
                self.rotation = self._keep[-1]
            ch, th = semkv_lloyd_max_gaussian(levels_hi)
            cl, tl = semkv_lloyd_max_gaussian(levels_lo)
            tabs = [t.to(device).contiguous() for t in (ch, th, cl, tl)]
            self._keep += tabs
            s.centroids_hi, s.thresholds_hi, s.centroids_lo, s.thresholds_lo = \
                [t.data_ptr() for t in tabs]
            self.codebooks = {"hi": (ch, th), "lo": (cl, tl)}
        elif base == BASE_AFFINE_HAD:
            assert signs is not None, "the rotated affine base needs a sign vector per (layer, head)"
            sg = torch.as_tensor(signs, dtype=torch.int8).to(device).contiguous()
            self._keep.append(sg)
            s.signs = sg.data_ptr()
            self.signs = sg
        self.s = s


def _round16(n: int) -> int:
    return (n + 15) // 16 * 16


class KVCache:
    """Owns the device buffers of one semkv_cache (torch allocations) and the
    struct the library reads and updates."""

    def __init__(self, desc: QuantDesc, batch: int, layers: int, kv_heads: int, q_heads: int,
                 hi_cap: int, lo_cap: int, block: int = 128, device="cuda"):
        self.desc = desc
        hi_cap, lo_cap = _round16(max(hi_cap, 16)), _round16(max(lo_cap, 16))
        rh = semkv_record_bytes(desc.base, desc.levels_hi)
        rl = semkv_record_bytes(desc.base, desc.levels_lo)
        dev = torch.device(device)
        u8 = dict(dtype=torch.uint8, device=dev)
        self.hi_pool = torch.zeros((batch, layers, kv_heads, hi_cap, rh), **u8)
        self.lo_pool = torch.zeros((batch, layers, kv_heads, lo_cap, rl), **u8)
        self.hi_tok = torch.full((batch, hi_cap), -1, dtype=torch.int32, device=dev)
        self.lo_tok = torch.full((batch, lo_cap), -1, dtype=torch.int32, device=dev)
        self.stage_k = torch.zeros((batch, layers, kv_heads, block, HEAD_DIM), dtype=torch.float16,
                                   device=dev)
        self.stage_v = torch.zeros_like(self.stage_k)
        self.stage_score = torch.zeros((batch, block), dtype=torch.float32, device=dev)
        self.blk_is_high = torch.zeros((batch, block), **u8)
        self.blk_slot = torch.zeros((batch, block), dtype=torch.int32, device=dev)
        self.dev_error = torch.zeros(1, dtype=torch.int32, device=dev)
        self.s = CacheStruct(batch=batch, layers=layers, kv_heads=kv_heads, q_heads=q_heads,
                             head_dim=HEAD_DIM, block=block,
                             hi_pool=self.hi_pool.data_ptr(), lo_pool=self.lo_pool.data_ptr(),
                             hi_cap=hi_cap, lo_cap=lo_cap, hi_tok=self.hi_tok.data_ptr(),
                             lo_tok=self.lo_tok.data_ptr(), hi_count=0, lo_count=0, n_tokens=0,
                             stage_k=self.stage_k.data_ptr(), stage_v=self.stage_v.data_ptr(),
                             stage_score=self.stage_score.data_ptr(), stage_n=0,
                             blk_is_high=self.blk_is_high.data_ptr(),
                             blk_slot=self.blk_slot.data_ptr(),
                             dev_error=self.dev_error.data_ptr())

    # host mirrors kept by the library
    @property
    def hi_count(self):
        return self.s.hi_count

    @property
    def lo_count(self):
        return self.s.lo_count

    @property
    def n_tokens(self):
        return self.s.n_tokens

    @property
    def stage_n(self):
        return self.s.stage_n

    def stage_token(self, k_tok: torch.Tensor, v_tok: torch.Tensor, score: torch.Tensor):
        """Algorithm 2: append a generated token at full precision and record its
        score (a device copy into staging slot stage_n; no per-token decision)."""
        n = self.s.stage_n
        if n >= self.s.block:
            raise SemkvError("stage_token", 3)
        self.stage_k[:, :, :, n].copy_(k_tok)
        self.stage_v[:, :, :, n].copy_(v_tok)
        self.stage_score[:, n].copy_(score)
        self.s.stage_n = n + 1

    def workspace(self):
        nbytes = semkv_decode_workspace_bytes(self)
        return torch.empty(nbytes // 4, dtype=torch.float32, device=self.hi_pool.device)
