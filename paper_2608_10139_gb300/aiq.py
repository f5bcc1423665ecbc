"""ctypes binding of libaiq.so: argument marshalling only.

Every step of a query runs in the library's CUDA kernels; this module only
turns numpy arrays and Python values into the C structs of ``include/aiq.h``
and ``include/aiq_ops.h`` and copies results back out.  It raises if the
compiled library is missing: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libaiq.so")

OK, ERR_INVALID_ARG, ERR_NOT_FOUND, ERR_OOM, ERR_CUDA, ERR_CAPACITY, ERR_DEVICE_CHECK, ERR_UNSUPPORTED = \
    0, -1, -2, -3, -4, -5, -6, -7
INT32, INT64, FLOAT32, TOKENS = 0, 1, 2, 3
LT, LE, GT, GE, EQ, NE = 0, 1, 2, 3, 4, 5
AGG_COUNT, AGG_ROW_IDS, AGG_GROUP_LABEL, AGG_GROUP_BUILD_KEY, AGG_SUM = 0, 1, 2, 3, 4
FLAG_LOGITS, FLAG_RELATIONAL_ONLY = 1, 2
GEN_MATCH_TOKENS = 1
EPI_F16, EPI_ROPE_F16, EPI_RESID_F32, EPI_SWIGLU_F16, EPI_RESID_ADD_F32 = 0, 1, 2, 3, 5


class AiqError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"aiq status {status}: {message}")
        self.status = status


class _Column(C.Structure):
    _fields_ = [("name", C.c_char_p), ("type", C.c_int32), ("data", C.c_void_p), ("offsets", C.c_void_p)]


class _ModelConfig(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("d_ffn", C.c_int32),
                ("vocab", C.c_int32), ("rope_theta", C.c_float), ("rms_eps", C.c_float)]


class _Pred(C.Structure):
    _fields_ = [("column", C.c_int32), ("op", C.c_int32), ("ivalue", C.c_int64), ("fvalue", C.c_double)]


class _Select(C.Structure):
    _fields_ = [("preds", C.POINTER(_Pred)), ("n_preds", C.c_int32), ("text_column", C.c_int32),
                ("prefix", C.POINTER(C.c_int32)), ("prefix_len", C.c_int32),
                ("label_ids", C.POINTER(C.c_int32)), ("n_labels", C.c_int32), ("agg", C.c_int32),
                ("flags", C.c_int32), ("sum_column", C.c_int32)]


class _View(C.Structure):
    _fields_ = [("n_input_rows", C.c_int64), ("n_candidates", C.c_int64), ("n_tokens", C.c_int64),
                ("n_chunks", C.c_int64), ("count", C.c_int64),
                ("row_ids", C.POINTER(C.c_int32)), ("n_row_ids", C.c_int64),
                ("group_build_rows", C.POINTER(C.c_int32)), ("group_keys", C.POINTER(C.c_int64)),
                ("group_counts", C.POINTER(C.c_int64)), ("n_groups", C.c_int64),
                ("label_counts", C.POINTER(C.c_int64)), ("n_labels", C.c_int32),
                ("cand_row_ids", C.POINTER(C.c_int32)), ("cand_build_rows", C.POINTER(C.c_int32)),
                ("label_logits", C.POINTER(C.c_float)), ("decisions", C.POINTER(C.c_int32)),
                ("ms_relational", C.c_float), ("ms_prefill", C.c_float), ("ms_aggregate", C.c_float),
                ("ms_total", C.c_float), ("prefill_flops", C.c_double), ("n_launches", C.c_int64),
                ("n_prefill_tokens", C.c_int64), ("row_ids_b", C.POINTER(C.c_int32)),
                ("gen_max_new", C.c_int32), ("n_gen_rows", C.c_int64), ("gen_row_ids", C.POINTER(C.c_int32)),
                ("gen_tokens", C.POINTER(C.c_int32)), ("gen_text_len", C.POINTER(C.c_int32)),
                ("ms_decode", C.c_float), ("decode_flops", C.c_double), ("n_decode_steps", C.c_int64),
                ("sum_int", C.c_int64), ("sum_float", C.c_double)]


class _Generate(C.Structure):
    _fields_ = [("max_new_tokens", C.c_int32), ("eos_id", C.c_int32), ("pad_id", C.c_int32),
                ("like_tokens", C.POINTER(C.c_int32)), ("like_len", C.c_int32), ("flags", C.c_int32)]


class _Term(C.Structure):
    _fields_ = [("column", C.c_void_p), ("type", C.c_int32), ("op", C.c_int32), ("ivalue", C.c_int64),
                ("fvalue", C.c_double)]


class _KStat(C.Structure):
    _fields_ = [("name", C.c_char_p), ("launches", C.c_int64), ("total_ms", C.c_double),
                ("flops", C.c_double), ("bytes", C.c_double)]


_lib = None

# (name, argtypes) of every exported entry point, mirroring the headers.
_SIGS = {
    "aiq_init": [C.c_int, C.POINTER(C.c_void_p)],
    "aiq_shutdown": [C.c_void_p],
    "aiq_load_table": [C.c_void_p, C.POINTER(_Column), C.c_int32, C.c_int64, C.POINTER(C.c_int64)],
    "aiq_free_table": [C.c_void_p, C.c_int64],
    "aiq_load_model": [C.c_void_p, C.POINTER(_ModelConfig), C.POINTER(C.c_void_p), C.c_int32, C.POINTER(C.c_int64)],
    "aiq_free_model": [C.c_void_p, C.c_int64],
    "aiq_run_select": [C.c_void_p, C.c_int64, C.c_int64, C.POINTER(_Select), C.POINTER(C.c_int64)],
    "aiq_run_join_select": [C.c_void_p, C.c_int64, C.c_int32, C.POINTER(_Pred), C.c_int32, C.c_int64, C.c_int32,
                            C.c_int64, C.POINTER(_Select), C.POINTER(C.c_int64)],
    "aiq_run_pair_select": [C.c_void_p, C.c_int64, C.c_int32, C.c_int64, C.POINTER(_Select), C.POINTER(C.c_int64)],
    "aiq_run_transform": [C.c_void_p, C.c_int64, C.c_int64, C.POINTER(_Select), C.POINTER(_Generate),
                          C.POINTER(C.c_int64)],
    "aiq_result": [C.c_void_p, C.c_int64, C.POINTER(_View)],
    "aiq_result_free": [C.c_void_p, C.c_int64],
    "aiq_last_error": [],
    "aiq_set_option": [C.c_void_p, C.c_char_p, C.c_int64],
    "aiq_stream": [C.c_void_p],
    "aiq_kernel_stats": [C.c_void_p, C.POINTER(_KStat), C.c_int32, C.POINTER(C.c_int32)],
    "aiq_reset_kernel_stats": [C.c_void_p],
    "aiq_op_gemm": [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_int64, C.c_int32, C.c_int32, C.c_int32,
                    C.c_int32, C.c_int32, C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                    C.c_int32],
    "aiq_op_rope_table": [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_float],
    "aiq_op_rmsnorm": [C.c_void_p, C.c_void_p, C.c_int64, C.c_int32, C.c_void_p, C.c_float, C.c_void_p],
    "aiq_op_attention": [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int32,
                         C.c_void_p, C.c_int32, C.c_void_p],
    "aiq_op_decode_attention": [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_void_p,
                                C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_void_p],
    "aiq_filter_compact_static": [C.POINTER(_Term), C.c_int32, C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p],
    "aiq_op_wait_expiry_selftest": [C.c_void_p, C.c_uint64],
}


def lib_path() -> str:
    return _LIB_PATH


def load_library():
    """Loads libaiq.so (built in-tree by ``build.py``); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"{_LIB_PATH} is not built; run paper_2608_10139_gb300.build.build() first")
    lib = C.CDLL(_LIB_PATH)
    for name, args in _SIGS.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = C.c_int
    lib.aiq_last_error.restype = C.c_char_p
    lib.aiq_shutdown.restype = None
    lib.aiq_stream.restype = C.c_void_p
    _lib = lib
    return lib


def _check(status: int):
    if status != OK:
        raise AiqError(status, _lib.aiq_last_error().decode())


def filter_compact_static(terms, n_rows: int, ids_out: int, count_out: int, stream: int = 0):
    """Allocation-free filter + compaction on device columns (see aiq_ops.h).
    terms: (device pointer, dtype code, op, constant) tuples; ids_out and
    count_out are device pointers; runs asynchronously on `stream`."""
    lib = load_library()
    ts = [_Term(p, t, op, int(v) if t != FLOAT32 else 0, float(v)) for p, t, op, v in terms]
    arr = (_Term * max(len(ts), 1))(*ts)
    _check(lib.aiq_filter_compact_static(arr, len(ts), n_rows, ids_out or None, count_out or None, stream or None))


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


@dataclass
class TableRef:
    handle: int
    n_rows: int
    names: List[str]
    types: List[int] = None

    def col(self, name: str) -> int:
        return self.names.index(name)


@dataclass
class Result:
    n_input_rows: int
    n_candidates: int
    n_tokens: int
    n_chunks: int
    count: int
    row_ids: np.ndarray
    group_build_rows: np.ndarray
    group_keys: np.ndarray
    group_counts: np.ndarray
    label_counts: np.ndarray
    cand_row_ids: np.ndarray
    cand_build_rows: np.ndarray
    label_logits: np.ndarray
    decisions: np.ndarray
    ms_relational: float
    ms_prefill: float
    ms_aggregate: float
    ms_total: float
    prefill_flops: float
    n_launches: int
    n_prefill_tokens: int
    row_ids_b: np.ndarray = None   # pair queries: B row of each yes pair
    sum: object = None             # AGG_SUM: int (integer column) or float


@dataclass
class TransformResult:
    n_input_rows: int
    n_candidates: int
    count: int                 # LIKE matches (-1 without LIKE)
    row_ids: np.ndarray        # LIKE: matching rows, ascending
    gen_row_ids: np.ndarray    # rows of gen_tokens
    gen_tokens: np.ndarray     # [n_gen_rows, max_new]
    gen_text_len: np.ndarray   # [n_gen_rows]
    ms_relational: float
    ms_prefill: float          # prefill and decode
    ms_decode: float
    ms_aggregate: float
    ms_total: float
    prefill_flops: float
    decode_flops: float
    n_decode_steps: int
    n_launches: int
    n_chunks: int


def _arr(ptr, n, dtype, shape=None):
    if n <= 0 or not ptr:
        return np.zeros(shape if shape is not None else (0,), dtype=dtype)
    a = np.ctypeslib.as_array(ptr, shape=(n,)).astype(dtype, copy=True)
    return a.reshape(shape) if shape is not None else a


class Context:
    """One library context on one CUDA device (its own stream and buffers)."""

    def __init__(self, device: int = 0):
        self._sum_float = False
        self._sum = None
        self.lib = load_library()
        h = C.c_void_p()
        _check(self.lib.aiq_init(device, C.byref(h)))
        self.h = h

    def close(self):
        if self.h:
            self.lib.aiq_shutdown(self.h)
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # --------------------------------------------------------------- tables
    def load_table(self, cols: Dict[str, np.ndarray], text: Optional[Tuple[np.ndarray, np.ndarray]] = None,
                   text_name: str = "text", n_rows: Optional[int] = None) -> TableRef:
        """cols: name -> int32 / int64 / float32 array; text: (int64 offsets [n+1], int32 ids)."""
        keep = []
        specs = []
        names = []
        types = []
        n = n_rows
        for name, a in cols.items():
            a = np.ascontiguousarray(a)
            t = {np.dtype(np.int32): INT32, np.dtype(np.int64): INT64, np.dtype(np.float32): FLOAT32}.get(a.dtype)
            if t is None:
                raise TypeError(f"column {name}: unsupported dtype {a.dtype}")
            n = len(a) if n is None else n
            keep.append(a)
            specs.append(_Column(name.encode(), t, a.ctypes.data, None))
            names.append(name)
            types.append(t)
        if text is not None:
            off = np.ascontiguousarray(text[0], dtype=np.int64)
            ids = _i32(text[1])
            n = len(off) - 1 if n is None else n
            keep += [off, ids]
            specs.append(_Column(text_name.encode(), TOKENS, ids.ctypes.data if ids.size else off.ctypes.data,
                                 off.ctypes.data))
            names.append(text_name)
            types.append(TOKENS)
        arr = (_Column * len(specs))(*specs)
        h = C.c_int64()
        _check(self.lib.aiq_load_table(self.h, arr, len(specs), n or 0, C.byref(h)))
        return TableRef(h.value, n or 0, names, types)

    def free_table(self, t: TableRef):
        _check(self.lib.aiq_free_table(self.h, t.handle))

    # --------------------------------------------------------------- models
    def load_model(self, shape, tensors: Sequence[np.ndarray]) -> int:
        """shape: object with n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ffn,
        vocab, rope_theta, rms_eps; tensors: bf16 bit patterns (uint16) in the
        documented order."""
        cfg = _ModelConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                           shape.d_ffn, shape.vocab, shape.rope_theta, shape.rms_eps)
        ts = [np.ascontiguousarray(t, dtype=np.uint16) for t in tensors]
        ptrs = (C.c_void_p * len(ts))(*[t.ctypes.data for t in ts])
        h = C.c_int64()
        _check(self.lib.aiq_load_model(self.h, C.byref(cfg), ptrs, len(ts), C.byref(h)))
        return h.value

    def free_model(self, m: int):
        _check(self.lib.aiq_free_model(self.h, m))

    # -------------------------------------------------------------- queries
    @staticmethod
    def _preds(t: TableRef, preds) -> Tuple[object, int]:
        ps = [_Pred(t.col(c), op, int(v), float(v)) for c, op, v in preds]
        arr = (_Pred * max(len(ps), 1))(*ps)
        return arr, len(ps)

    def _select(self, t: TableRef, preds, prefix, labels, agg, flags, text_name, sum_column=None):
        parr, np_ = self._preds(t, preds)
        prefix = _i32(prefix)
        labels = _i32(labels)
        sel = _Select(parr, np_, t.col(text_name) if text_name in t.names else -1,
                      prefix.ctypes.data_as(C.POINTER(C.c_int32)), len(prefix),
                      labels.ctypes.data_as(C.POINTER(C.c_int32)), len(labels), agg, flags,
                      t.col(sum_column) if sum_column is not None else -1)
        return sel, (parr, prefix, labels)

    def _fetch(self, h: C.c_int64, k: int) -> Result:
        v = _View()
        try:
            _check(self.lib.aiq_result(self.h, h, C.byref(v)))
            s = v.n_candidates
            self._sum = v.sum_float if self._sum_float else v.sum_int
            return Result(
                v.n_input_rows, v.n_candidates, v.n_tokens, v.n_chunks, v.count,
                _arr(v.row_ids, v.n_row_ids, np.int32),
                _arr(v.group_build_rows, v.n_groups, np.int32),
                _arr(v.group_keys, v.n_groups, np.int64),
                _arr(v.group_counts, v.n_groups, np.int64),
                _arr(v.label_counts, v.n_labels, np.int64),
                _arr(v.cand_row_ids, s if v.cand_row_ids else 0, np.int32),
                _arr(v.cand_build_rows, s if v.cand_build_rows else 0, np.int32),
                _arr(v.label_logits, s * k if v.label_logits else 0, np.float32,
                     (s, k) if v.label_logits else (0, k)),
                _arr(v.decisions, s if v.decisions else 0, np.int32),
                v.ms_relational, v.ms_prefill, v.ms_aggregate, v.ms_total, v.prefill_flops, v.n_launches,
                v.n_prefill_tokens, _arr(v.row_ids_b, v.n_row_ids if v.row_ids_b else 0, np.int32),
                self._sum)
        finally:
            self.lib.aiq_result_free(self.h, h)

    def run_select(self, table: TableRef, model: int, preds, prefix, labels, agg: int = AGG_COUNT,
                   flags: int = 0, text_name: str = "text", sum_column: Optional[str] = None) -> Result:
        """preds: (column name, op, constant) triples, conjoined.  AGG_SUM sums
        ``sum_column`` over the yes rows (Result.sum: int, or float for a FLOAT32 column)."""
        self._sum_float = sum_column is not None and table.types[table.col(sum_column)] == FLOAT32
        sel, keep = self._select(table, preds, prefix, labels, agg, flags, text_name, sum_column)
        h = C.c_int64()
        _check(self.lib.aiq_run_select(self.h, table.handle, model, C.byref(sel), C.byref(h)))
        return self._fetch(h, len(labels))

    def run_join_select(self, build: TableRef, build_key: str, build_preds, probe: TableRef, probe_key: str,
                        model: int, preds, prefix, labels, agg: int = AGG_GROUP_BUILD_KEY, flags: int = 0,
                        text_name: str = "text") -> Result:
        bparr, nbp = self._preds(build, build_preds)
        self._sum_float = False
        sel, keep = self._select(probe, preds, prefix, labels, agg, flags, text_name)
        h = C.c_int64()
        _check(self.lib.aiq_run_join_select(self.h, build.handle, build.col(build_key), bparr, nbp, probe.handle,
                                            probe.col(probe_key), model, C.byref(sel), C.byref(h)))
        return self._fetch(h, len(labels))

    def run_pair_select(self, table: TableRef, key: str, model: int, preds, prefix, labels,
                        agg: int = AGG_ROW_IDS, flags: int = 0, text_name: str = "text") -> Result:
        """Table 2 Q4: AI_IF over every (a < b) pair of selected rows with equal ``key``;
        candidates are the pairs (cand_row_ids / cand_build_rows = A / B rows)."""
        self._sum_float = False
        sel, keep = self._select(table, preds, prefix, labels, agg, flags, text_name)
        h = C.c_int64()
        _check(self.lib.aiq_run_pair_select(self.h, table.handle, table.col(key), model, C.byref(sel), C.byref(h)))
        return self._fetch(h, len(labels))

    def run_transform(self, table: TableRef, model: int, preds, prefix, max_new: int, eos: int = -1,
                      pad: int = 0, like=None, match_tokens: bool = False,
                      text_name: str = "text") -> TransformResult:
        """AI_TRANSFORM (greedy) of every candidate row; with ``like`` (a token
        sequence) only the COUNT / ids of the rows whose output contains it."""
        sel, keep = self._select(table, preds, prefix, [], AGG_COUNT, 0, text_name)
        pat = _i32(like if like is not None else [])
        buf = pat if pat.size else np.zeros(1, np.int32)   # a non-NULL pointer for the empty pattern
        g = _Generate(max_new, eos, pad,
                      buf.ctypes.data_as(C.POINTER(C.c_int32)) if like is not None else None,
                      len(pat), GEN_MATCH_TOKENS if match_tokens else 0)
        h = C.c_int64()
        _check(self.lib.aiq_run_transform(self.h, table.handle, model, C.byref(sel), C.byref(g), C.byref(h)))
        v = _View()
        try:
            _check(self.lib.aiq_result(self.h, h, C.byref(v)))
            n, w = v.n_gen_rows, v.gen_max_new
            return TransformResult(
                v.n_input_rows, v.n_candidates, v.count, _arr(v.row_ids, v.n_row_ids, np.int32),
                _arr(v.gen_row_ids, n, np.int32),
                _arr(v.gen_tokens, n * w, np.int32, (n, w)) if n else np.zeros((0, w), np.int32),
                _arr(v.gen_text_len, n, np.int32),
                v.ms_relational, v.ms_prefill, v.ms_decode, v.ms_aggregate, v.ms_total, v.prefill_flops,
                v.decode_flops, v.n_decode_steps, v.n_launches, v.n_chunks)
        finally:
            self.lib.aiq_result_free(self.h, h)

    # -------------------------------------------------------------- options
    def set_option(self, name: str, value: int):
        _check(self.lib.aiq_set_option(self.h, name.encode(), int(value)))

    def stream(self) -> int:
        return self.lib.aiq_stream(self.h) or 0

    def kernel_stats(self) -> Dict[str, dict]:
        buf = (_KStat * 64)()
        n = C.c_int32()
        _check(self.lib.aiq_kernel_stats(self.h, buf, 64, C.byref(n)))
        return {buf[i].name.decode(): dict(launches=buf[i].launches, total_ms=buf[i].total_ms,
                                           flops=buf[i].flops, bytes=buf[i].bytes) for i in range(n.value)}

    def reset_kernel_stats(self):
        _check(self.lib.aiq_reset_kernel_stats(self.h))

    # ------------------------------------------------- step-level (device ptrs)
    def op_gemm(self, A: int, lda: int, B: int, ldb: int, M: int, N: int, K: int, bn: int, epilogue: int,
                out: int, ldo: int, positions: int = 0, rope_cos: int = 0, rope_sin: int = 0,
                rope_cols: int = 0, head_dim: int = 0):
        _check(self.lib.aiq_op_gemm(self.h, A, lda, B, ldb, M, N, K, bn, epilogue, out, ldo, positions or None,
                                    rope_cos or None, rope_sin or None, rope_cols, head_dim))

    def op_rope_table(self, cos_ptr: int, sin_ptr: int, max_pos: int, head_dim: int, theta: float):
        _check(self.lib.aiq_op_rope_table(self.h, cos_ptr, sin_ptr, max_pos, head_dim, theta))

    def op_rmsnorm(self, x: int, T: int, d: int, g: int, eps: float, out: int):
        _check(self.lib.aiq_op_rmsnorm(self.h, x, T, d, g, eps, out))

    def op_attention(self, qkv: int, T: int, seq_start: int, n_seqs: int, Hq: int, Hkv: int, hd: int, out: int,
                     prefix_kv: int = 0, P: int = 0):
        _check(self.lib.aiq_op_attention(self.h, qkv, T, seq_start, n_seqs, Hq, Hkv, hd, prefix_kv or None, P, out))

    def op_wait_expiry_selftest(self, limit_ns: int):
        """Runs the bounded-wait self-test (see aiq_ops.h); raises AiqError
        with AIQ_ERR_DEVICE_CHECK when the wait expired as it should."""
        _check(self.lib.aiq_op_wait_expiry_selftest(self.h, limit_ns))

    def op_decode_attention(self, qkv: int, R: int, Hq: int, Hkv: int, hd: int, own_kv: int, seq_start: int,
                            gen_kv: int, gen_cap: int, slot: int, out: int, prefix_kv: int = 0, P: int = 0):
        _check(self.lib.aiq_op_decode_attention(self.h, qkv, R, Hq, Hkv, hd, prefix_kv or None, P, own_kv, seq_start,
                                                gen_kv, gen_cap, slot, out))
