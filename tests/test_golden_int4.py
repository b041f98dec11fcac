"""The stored oracle values of the 80-block int4 workload (tests/golden/int4_72B_80L_step0.npz):
written by tests/golden/make_int4_72B_goldens.py, which calls only the oracle and the seeded
generator.  Checked here without a GPU: the file records the script that wrote it, its inputs are
the workload generator's, and its parts agree with one another."""
import hashlib
import os

import numpy as np
import pytest

from paper_2609_34045_gb300 import workload as wl

HERE = os.path.dirname(os.path.abspath(__file__))
GOLDEN = os.path.join(HERE, "golden", "int4_72B_80L_step0.npz")
SCRIPT = os.path.join(HERE, "golden", "make_int4_72B_goldens.py")


@pytest.fixture(scope="module")
def gold():
    return np.load(GOLDEN)


def test_written_by_the_committed_script(gold):
    with open(SCRIPT, "rb") as f:
        assert str(gold["script_sha256"]) == hashlib.sha256(f.read()).hexdigest()
    assert len(str(gold["oracle_sha256"])) == 64


def test_inputs_are_the_generators(gold):
    w = wl.CONFIGS[6]
    assert int(gold["seed"]) == w.seed == wl.CONFIGS[5].seed
    assert np.array_equal(gold["positions"], wl.positions(w, 0))
    assert np.array_equal(gold["token_ids"], wl.first_token_ids(w.model, 4, w.seed))
    # batch one is user 0 of the batch: the same first token and position
    assert np.array_equal(wl.first_token_ids(w.model, 1, w.seed), gold["token_ids"][:1])
    cols = gold["sample_cols"]
    assert cols.size == 512 and np.all(np.diff(cols) > 0) and cols[-1] < w.model.d_model


def test_parts_agree(gold):
    cols = gold["sample_cols"]
    rms = gold["per_layer_rms"]
    assert rms.shape == (80, 4) and np.all(np.isfinite(rms)) and np.all(rms > 0)
    for i, n in enumerate(gold["full_layers"]):
        full = gold["full_states"][i].astype(np.float64)
        assert np.allclose(np.sqrt(np.mean(full * full, axis=-1)), rms[n - 1], rtol=1e-6)
        assert np.array_equal(gold["full_states"][i][:, cols], gold["per_layer_sample"][n - 1])
    top, z = gold["top_ids"], gold["top_logits"]
    assert np.all(np.diff(z, axis=-1) <= 0)
    assert np.array_equal(gold["next_ids"], top[:, 0])
    assert np.allclose(gold["margins"], z[:, 0] - z[:, 1])
    assert gold["k_new"].shape == gold["v_new"].shape == (6, 4, 8, 128)
