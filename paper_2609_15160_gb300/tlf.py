"""ctypes binding of libtlf (include/tlf.h): argument marshalling only.

Module-level functions carry the C names (``tlf_create``, ``tlf_prefill``,
``tlf_decode_step``, ``tlf_release``, ...). ``Context`` wraps them for
numpy / torch callers. Every computation of the decode step runs in the CUDA
kernels of libtlf; when the library has not been built this module raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import build as _build
from . import synth as _synth

TLF_OK = 0
ERRORS = {-1: "INVALID_ARG", -2: "UNKNOWN_SEQ", -3: "DUPLICATE_SEQ", -4: "OUT_OF_PAGES", -5: "SEQ_TOO_LONG",
          -6: "CUDA", -7: "BAD_WEIGHTS", -8: "DEVICE", -9: "NO_DEVICE", -10: "CAPACITY"}
CODES = {v: k for k, v in ERRORS.items()}
KERNEL_CLASSES = ("router", "plan", "attn_norm", "qkv_gemm", "rope_append", "attention", "o_gemm", "mlp_norm",
                  "gate_up_gemm", "swiglu", "down_gemm", "final_norm", "lm_head")
DTYPE = {"f32": 0, "bf16": 1}
EXIT = {"argmax": 0, "survival": 1}
GEMM = {"auto": 0, "simt": 1}
ABLATION = {"none": 0, "no_gather": 1, "dense_cache": 2}


class TlfConfig(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("vocab", "d_model", "n_heads", "n_kv_heads", "head_dim", "n_layers",
                                         "ffn_hidden", "max_loops")] + [
        ("rope_base", C.c_float), ("norm_eps", C.c_float), ("dtype", C.c_int32), ("exit_rule", C.c_int32),
        ("threshold", C.c_float), ("max_seqs", C.c_int32), ("max_batch", C.c_int32), ("max_seq_len", C.c_int32),
        ("page_size", C.c_int32), ("gemm_impl", C.c_int32), ("host_only", C.c_int32), ("prefill_chunk", C.c_int32),
        ("kv_pool_pages", C.c_int64), ("ablation", C.c_int32), ("conditioning", C.c_int32),
        ("router_hidden", C.c_int32), ("reserved", C.c_int32)]


COND_WEIGHTS = ("cond_t_w1", "cond_t_b1", "cond_t_w2", "cond_t_b2", "cond_dt_w1", "cond_dt_b1", "cond_dt_w2",
                "cond_dt_b2", "mod_w", "mod_b")


class TlfWeights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("embedding", "router_w", "router_b", "wq", "wk", "wv", "wo", "w_gate",
                                          "w_up", "w_down", "attn_norm", "mlp_norm", "final_norm") + COND_WEIGHTS
                + ("router_w1", "router_b1")]


class TlfAttnArgs(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("n", "n_heads", "n_kv_heads", "head_dim", "n_layers", "layer",
                                         "page_size", "dtype", "max_pages", "reserved0")] + [
        ("n_pages", C.c_int64)] + [(n, C.c_void_p) for n in ("q", "pool", "page_table", "lens", "out", "err")]


class TlfError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERRORS.get(code, code)}: {msg}")
        self.code = code
        self.name = ERRORS.get(code, str(code))


_LIB = None
_P = C.c_void_p
_I32P = C.POINTER(C.c_int32)
_U64P = C.POINTER(C.c_uint64)
_F32P = C.POINTER(C.c_float)

_SIGS = {
    "tlf_validate_config": (C.c_int, [C.POINTER(TlfConfig), C.c_char_p, C.c_size_t]),
    "tlf_page_bytes": (C.c_int64, [C.POINTER(TlfConfig)]),
    "tlf_create": (C.c_int, [C.POINTER(TlfConfig), C.POINTER(TlfWeights), C.POINTER(_P)]),
    "tlf_destroy": (None, [_P]),
    "tlf_last_error": (C.c_char_p, [_P]),
    "tlf_prefill": (C.c_int, [_P, C.c_int32, _U64P, _I32P, _I32P, _I32P, _P, _I32P, _P]),
    "tlf_decode_step": (C.c_int, [_P, C.c_int32, _U64P, _I32P, _I32P, _P, _I32P, _F32P, _P]),
    "tlf_release": (C.c_int, [_P, C.c_uint64]),
    "tlf_load_cache": (C.c_int, [_P, C.c_uint64, _I32P, _I32P, _P, _P]),
    "tlf_stats": (C.c_int, [_P, _I32P, C.POINTER(C.c_int64), C.POINTER(C.c_int64)]),
    "tlf_cache_len": (C.c_int, [_P, C.c_uint64, C.c_int32, _I32P]),
    "tlf_read_cache": (C.c_int, [_P, C.c_uint64, C.c_int32, C.c_int32, _I32P, _F32P, _F32P]),
    "tlf_last_active_sets": (C.c_int, [_P, _I32P, _I32P]),
    "tlf_set_profiling": (C.c_int, [_P, C.c_int32]),
    "tlf_last_step_profile": (C.c_int, [_P, _F32P, C.POINTER(C.c_double), _I32P]),
    "tlf_last_step_kernel_times": (C.c_int, [_P, _F32P, C.c_int32]),
    "tlf_attn_decode_scratch_bytes": (C.c_size_t, [C.POINTER(TlfAttnArgs)]),
    "tlf_attn_decode": (C.c_int, [C.POINTER(TlfAttnArgs), _P, C.c_size_t, _P]),
    "tlf_attn_decode_static": (C.c_int, [C.POINTER(TlfAttnArgs), _P]),
}


def library_path() -> str:
    return _build.LIB


def load_library(path: Optional[str] = None):
    """Load libtlf.so (built in-tree by __graft_entry__.build()); raises if missing."""
    global _LIB
    if _LIB is not None and path is None:
        return _LIB
    p = path or library_path()
    if not os.path.exists(p):
        raise RuntimeError(f"libtlf.so not found at {p}: build it with __graft_entry__.build() "
                           "(the decode step has no fallback path)")
    lib = C.CDLL(p)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _LIB = lib
    return lib


def _ptr(a, ctype):
    return None if a is None else a.ctypes.data_as(C.POINTER(ctype))


def _check(rc: int, ctx=None):
    if rc != TLF_OK:
        msg = load_library().tlf_last_error(ctx).decode()
        raise TlfError(rc, msg)


def _addr(buf) -> Optional[int]:
    """Address of a numpy array or a torch tensor (host or device)."""
    if buf is None:
        return None
    if hasattr(buf, "data_ptr"):
        return buf.data_ptr()
    return buf.ctypes.data


def _stream(stream) -> Optional[int]:
    if stream is None:
        return None
    if hasattr(stream, "cuda_stream"):
        return stream.cuda_stream
    return int(stream)


# ----------------------------------------------------------------------------
# C names
# ----------------------------------------------------------------------------

def make_config(m, max_seqs: int, max_batch: int, max_seq_len: int, page_size: int = 64,
                kv_pool_pages: int = 0, gemm_impl: str = "auto", host_only: bool = False,
                prefill_chunk: int = 0, ablation: str = "none") -> TlfConfig:
    return TlfConfig(vocab=m.vocab, d_model=m.d_model, n_heads=m.n_heads, n_kv_heads=m.n_kv_heads,
                     head_dim=m.head_dim, n_layers=m.n_layers, ffn_hidden=m.ffn_hidden, max_loops=m.max_loops,
                     rope_base=m.rope_base, norm_eps=m.norm_eps, dtype=DTYPE[m.dtype], exit_rule=EXIT[m.exit_rule],
                     threshold=m.threshold, max_seqs=max_seqs, max_batch=max_batch, max_seq_len=max_seq_len,
                     page_size=page_size, gemm_impl=GEMM[gemm_impl], host_only=int(host_only), prefill_chunk=prefill_chunk,
                     kv_pool_pages=kv_pool_pages, ablation=ABLATION[ablation],
                     conditioning=int(getattr(m, "conditioning", False)),
                     router_hidden=int(getattr(m, "router_hidden", 0)))


def tlf_validate_config(cfg: TlfConfig):
    buf = C.create_string_buffer(256)
    rc = load_library().tlf_validate_config(C.byref(cfg), buf, 256)
    return rc, buf.value.decode()


def tlf_page_bytes(cfg: TlfConfig) -> int:
    return load_library().tlf_page_bytes(C.byref(cfg))


def _matrix(a: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return np.ascontiguousarray(_synth.bf16_bits(a))
    return np.ascontiguousarray(a, dtype=np.float32)


def tlf_create(cfg: TlfConfig, weights: Optional[Dict[str, np.ndarray]], dtype: str):
    """Returns (ctx handle, kept arrays). weights: the dict of synth.make_weights."""
    keep = {}
    w = TlfWeights()
    if weights is not None:
        for name in ("embedding", "router_w", "wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down"):
            keep[name] = _matrix(weights[name], dtype)
        for name in ("router_b", "attn_norm", "mlp_norm", "final_norm"):
            keep[name] = np.ascontiguousarray(weights[name], dtype=np.float32)
        if cfg.conditioning:
            for name in COND_WEIGHTS:
                keep[name] = np.ascontiguousarray(weights[name], dtype=np.float32)
        if cfg.router_hidden:
            keep["router_w1"] = _matrix(weights["router_w1"], dtype)
            keep["router_b1"] = np.ascontiguousarray(weights["router_b1"], dtype=np.float32)
        for name, arr in keep.items():
            setattr(w, name, arr.ctypes.data)
    h = _P()
    rc = load_library().tlf_create(C.byref(cfg), C.byref(w) if weights is not None else None, C.byref(h))
    _check(rc, None)
    return h, keep


def tlf_destroy(ctx):
    load_library().tlf_destroy(ctx)


def tlf_prefill(ctx, seq_ids: np.ndarray, offsets: np.ndarray, tokens: np.ndarray, forced, last_logits, loops,
                stream=None):
    rc = load_library().tlf_prefill(ctx, len(seq_ids), _ptr(seq_ids, C.c_uint64), _ptr(offsets, C.c_int32),
                                    _ptr(tokens, C.c_int32), _ptr(forced, C.c_int32), _addr(last_logits),
                                    _ptr(loops, C.c_int32), _stream(stream))
    _check(rc, ctx)


def tlf_decode_step(ctx, seq_ids: np.ndarray, tokens: np.ndarray, forced, logits, loops: np.ndarray, margin,
                    stream=None):
    rc = load_library().tlf_decode_step(ctx, len(seq_ids), _ptr(seq_ids, C.c_uint64), _ptr(tokens, C.c_int32),
                                        _ptr(forced, C.c_int32), _addr(logits), _ptr(loops, C.c_int32),
                                        _ptr(margin, C.c_float), _stream(stream))
    _check(rc, ctx)


def tlf_release(ctx, seq_id: int):
    _check(load_library().tlf_release(ctx, C.c_uint64(seq_id)), ctx)


def tlf_load_cache(ctx, seq_id: int, lens: np.ndarray, positions: np.ndarray, k: Optional[np.ndarray],
                   v: Optional[np.ndarray]):
    """k = v = None: entries are filled on the device (see include/tlf.h)."""
    _check(load_library().tlf_load_cache(ctx, C.c_uint64(seq_id), _ptr(lens, C.c_int32), _ptr(positions, C.c_int32),
                                         None if k is None else k.ctypes.data,
                                         None if v is None else v.ctypes.data), ctx)


def attn_args(n, n_heads, n_kv_heads, head_dim, n_layers, layer, dtype, max_pages, n_pages, q, pool, page_table,
              lens, out, err=None) -> TlfAttnArgs:
    """Arguments of tlf_attn_decode; buffers are torch CUDA tensors (or raw device addresses)."""
    return TlfAttnArgs(n=n, n_heads=n_heads, n_kv_heads=n_kv_heads, head_dim=head_dim, n_layers=n_layers,
                       layer=layer, page_size=64, dtype=DTYPE[dtype] if isinstance(dtype, str) else dtype,
                       max_pages=max_pages, reserved0=0, n_pages=n_pages, q=_addr(q), pool=_addr(pool),
                       page_table=_addr(page_table), lens=_addr(lens), out=_addr(out), err=_addr(err))


def tlf_attn_decode_scratch_bytes(a: TlfAttnArgs) -> int:
    return load_library().tlf_attn_decode_scratch_bytes(C.byref(a))


def tlf_attn_decode(a: TlfAttnArgs, scratch, scratch_bytes: int, stream=None):
    _check(load_library().tlf_attn_decode(C.byref(a), _addr(scratch), scratch_bytes, _stream(stream)), None)


def tlf_attn_decode_static(a: TlfAttnArgs, stream=None):
    """tlf_attn_decode without caller scratch: uses the library's built-in 4 MiB device array."""
    _check(load_library().tlf_attn_decode_static(C.byref(a), _stream(stream)), None)


# ----------------------------------------------------------------------------
# convenience wrapper
# ----------------------------------------------------------------------------

class Context:
    """One library context for a model configuration (synth.ModelConfig)."""

    def __init__(self, model, weights: Optional[Dict[str, np.ndarray]], max_seqs: int, max_batch: int,
                 max_seq_len: int, kv_pool_pages: int = 0, gemm_impl: str = "auto", host_only: bool = False,
                 prefill_chunk: int = 0, ablation: str = "none"):
        self.model = model
        self.cfg = make_config(model, max_seqs, max_batch, max_seq_len, kv_pool_pages=kv_pool_pages,
                               gemm_impl=gemm_impl, host_only=host_only, prefill_chunk=prefill_chunk,
                               ablation=ablation)
        self.handle, _ = tlf_create(self.cfg, weights, model.dtype)
        self.max_batch = max_batch

    def close(self):
        if self.handle:
            tlf_destroy(self.handle)
            self.handle = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def prefill(self, seq_ids: Sequence[int], prompts: Sequence[np.ndarray], forced=None, logits: bool = True,
                logits_out=None, stream=None):
        """Returns (last logits [n, V] numpy or logits_out, loops list of int32 arrays)."""
        ids = np.asarray(seq_ids, dtype=np.uint64)
        lens = np.array([len(p) for p in prompts], dtype=np.int64)
        offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        toks = np.ascontiguousarray(np.concatenate([np.asarray(p, dtype=np.int32) for p in prompts]))
        frc = None if forced is None else np.ascontiguousarray(np.concatenate(
            [np.asarray(f, dtype=np.int32) for f in forced]))
        out = logits_out
        if logits and out is None:
            out = np.zeros((len(prompts), self.model.vocab), dtype=np.float32)
        loops = np.zeros(int(offsets[-1]), dtype=np.int32)
        tlf_prefill(self.handle, ids, offsets, toks, frc, out if logits else None, loops, stream)
        return out, [loops[offsets[i]:offsets[i + 1]] for i in range(len(prompts))]

    def decode_step(self, seq_ids: Sequence[int], tokens: Sequence[int], forced=None, logits=True, stream=None):
        """Returns (logits [B, V] (numpy, or the given buffer), loops [B], margins [B])."""
        ids = np.asarray(seq_ids, dtype=np.uint64)
        toks = np.ascontiguousarray(tokens, dtype=np.int32)
        frc = None if forced is None else np.ascontiguousarray(forced, dtype=np.int32)
        if logits is True:
            out = np.zeros((len(ids), self.model.vocab), dtype=np.float32)
        elif logits is False or logits is None:
            out = None
        else:
            out = logits
        loops = np.zeros(len(ids), dtype=np.int32)
        margin = np.zeros(len(ids), dtype=np.float32)
        tlf_decode_step(self.handle, ids, toks, frc, out, loops, margin, stream)
        return out, loops, margin

    def release(self, seq_id: int):
        tlf_release(self.handle, seq_id)

    def load_cache(self, seq_id: int, snapshot: dict):
        """snapshot: synth.make_cache_snapshot output (values exact in the model dtype); without
        "k"/"v" entries (synth.make_cache_positions) the values are filled on the device."""
        lens = np.array([len(p) for p in snapshot["positions"]], dtype=np.int32)
        pos = np.ascontiguousarray(np.concatenate(snapshot["positions"]).astype(np.int32))
        if "k" not in snapshot:
            tlf_load_cache(self.handle, seq_id, lens, pos, None, None)
            return
        k = np.concatenate(snapshot["k"]).astype(np.float32)
        v = np.concatenate(snapshot["v"]).astype(np.float32)
        tlf_load_cache(self.handle, seq_id, lens, pos, _matrix(k, self.model.dtype), _matrix(v, self.model.dtype))

    def stats(self):
        live, free, total = C.c_int32(), C.c_int64(), C.c_int64()
        _check(load_library().tlf_stats(self.handle, C.byref(live), C.byref(free), C.byref(total)), self.handle)
        return live.value, free.value, total.value

    def cache_len(self, seq_id: int, loop: int) -> int:
        n = C.c_int32()
        _check(load_library().tlf_cache_len(self.handle, C.c_uint64(seq_id), loop, C.byref(n)), self.handle)
        return n.value

    def read_cache(self, seq_id: int, loop: int, layer: int):
        n = self.cache_len(seq_id, loop)
        m = self.model
        pos = np.zeros(n, dtype=np.int32)
        k = np.zeros((n, m.n_kv_heads, m.head_dim), dtype=np.float32)
        v = np.zeros_like(k)
        _check(load_library().tlf_read_cache(self.handle, C.c_uint64(seq_id), loop, layer, _ptr(pos, C.c_int32),
                                             _ptr(k, C.c_float), _ptr(v, C.c_float)), self.handle)
        return pos, k, v

    def last_active_sets(self, batch: int):
        M = self.model.max_loops
        counts = np.zeros(M, dtype=np.int32)
        idx = np.zeros(M * batch, dtype=np.int32)
        _check(load_library().tlf_last_active_sets(self.handle, _ptr(counts, C.c_int32), _ptr(idx, C.c_int32)),
               self.handle)
        return counts, [idx[r * batch: r * batch + counts[r]] for r in range(M)]

    def set_profiling(self, on: bool):
        _check(load_library().tlf_set_profiling(self.handle, int(on)), self.handle)

    def last_step_profile(self):
        ms, by, nl = C.c_float(), C.c_double(), C.c_int32()
        _check(load_library().tlf_last_step_profile(self.handle, C.byref(ms), C.byref(by), C.byref(nl)), self.handle)
        return ms.value, by.value, nl.value

    def last_step_kernel_times(self) -> Dict[str, float]:
        """Milliseconds per kernel class of the last profiled step."""
        ms = np.zeros(len(KERNEL_CLASSES), dtype=np.float32)
        _check(load_library().tlf_last_step_kernel_times(self.handle, _ptr(ms, C.c_float), len(ms)), self.handle)
        return dict(zip(KERNEL_CLASSES, ms.tolist()))
