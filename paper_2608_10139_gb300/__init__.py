"""Unified AI-query execution on one GB300 (sm_103a).

The query pipeline (predicate, compaction, hash join, token packing, decoder
prefill, label decision, aggregate) lives in ``libaiq.so`` (CUDA, built from
``csrc/`` by ``build.py``); ``aiq`` is its ctypes binding.
"""
from . import aiq  # noqa: F401
from .aiq import AiqError, Context, Result, TableRef, load_library  # noqa: F401
