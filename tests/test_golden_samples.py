"""The stored oracle samples (tests/golden/oracle_logits_<workload>.json) are
consistent with the oracle as it stands: keyed by the current oracle and
input-generator sources, their rows are the oracle's own candidates at the
stored positions, and a stored row's label logits are what the oracle
computes for it here (checked on the shortest prompt of each 1B-shape sample;
the 8B weights are too large for the CPU suite)."""
import glob
import importlib.util
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
FILES = sorted(glob.glob(os.path.join(GOLDEN, "oracle_logits_*.json")))


def _mod():
    spec = importlib.util.spec_from_file_location("make_oracle_samples",
                                                  os.path.join(GOLDEN, "make_oracle_samples.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_stored_samples_exist_for_the_select_and_join_workloads():
    names = {os.path.basename(f)[len("oracle_logits_"):-len(".json")] for f in FILES}
    assert {"c2_select_1b", "c3_join_1b"} <= names


@pytest.mark.parametrize("path", FILES, ids=[os.path.basename(f) for f in FILES])
def test_stored_sample_matches_the_oracle(path):
    import synth
    from oracle import query as oq
    from oracle import transformer as tf
    mod = _mod()
    with open(path) as fh:
        d = json.load(fh)
    w = mod.workload(d["workload"])
    key = mod.key_of(w, d["sample_k"])
    assert all(d[k] == v for k, v in key.items()), "stale sample: rerun make_oracle_samples.py"
    q = synth.make_inputs(w)
    cand, _ = mod.candidates(w, q)
    pos = np.asarray(d["positions"], np.int64)
    assert d["n_candidates"] == len(cand)
    assert np.all(np.diff(pos) > 0) and pos[0] >= 0 and pos[-1] < len(cand)
    lens = np.diff(q.table.offsets)[cand]
    assert np.array_equal(pos, mod.sample_positions(len(cand), d["sample_k"], d["sample_seed"], lens))
    assert np.array_equal(np.asarray(d["row_ids"]), cand[pos])
    z = np.asarray(d["logits"], np.float64)
    assert z.shape == (len(pos), len(w.label_ids)) and np.isfinite(z).all()
    assert d["prompt_lens"] == [int(len(q.prefix) + lens[p]) for p in pos]
    if w.model.d_model <= 2048:
        i = int(np.argmin(d["prompt_lens"]))
        model = tf.Model(w.model, synth.make_weights(w.model, w.weight_seed))
        live = tf.label_logits(model, oq.prompts(q.prefix, q.table.offsets, q.table.tokens, [d["row_ids"][i]]),
                               w.label_ids)
        np.testing.assert_allclose(live[0], z[i], rtol=1e-9, atol=1e-9)
