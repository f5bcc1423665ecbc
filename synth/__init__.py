"""Seeded synthetic inputs shared by the oracle, the tests and the benchmark.

This package generates tables, prompt prefixes and random-init bf16 weights.
It contains no part of the query's arithmetic.
"""
from .configs import *  # noqa: F401,F403
from .generate import (QueryInputs, Table, bf16_bits_to_f32, distinct_int63,  # noqa: F401
                       f32_to_bf16_bits, make_inputs, make_join_inputs, make_pair_inputs,
                       make_select_inputs, make_weights, text_lengths,
                       weight_specs, zipf_ranks)
