"""Stored oracle values (``tests/golden/oracle_builds.json``, written by
``tests/golden/make_golden.py`` from the fp64 oracle alone).

On the CPU the fixture locks the oracle: a change of its arithmetic that moves a stored value
fails here and has to come with a regenerated fixture. On the GPU the CUDA build of the same
seeded inputs is compared with the stored values, so the device path is checked against
numbers that were fixed before it ran. The pins that tie the oracle to the paper are in
``test_oracle_pins.py``; these values add no pin of their own.
"""
import json
import os

import numpy as np
import pytest

import oracle
import synth
from tests.golden.make_golden import input_digest, sample

FIXTURE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "oracle_builds.json")


def _cases():
    with open(FIXTURE) as f:
        doc = json.load(f)
    out = []
    for c in doc["cases"]:
        fields = dict(c["config"])
        fields["mrope_section"] = tuple(fields["mrope_section"])
        fields["grid"] = tuple(fields["grid"])
        out.append((c, synth.Config(**fields)))
    return out


CASES = _cases()
IDS = [c["name"] for c, _ in CASES]


def _scaled_err(val, rms, ref_val, ref_rms):
    ref_val, ref_rms = np.asarray(ref_val), np.asarray(ref_rms)
    return float(np.max(np.abs(val - ref_val) / np.maximum(np.abs(ref_val), ref_rms[..., None])))


@pytest.mark.parametrize("case,cfg", CASES, ids=IDS)
def test_oracle_reproduces_stored_values(case, cfg):
    inp = synth.make_inputs(cfg)
    assert input_digest(inp) == case["inputs_sha256"], "the seeded input generator changed"
    ref = oracle.build_tokens(inp, np.asarray(case["tokens"]))
    k_rms, k = sample(cfg, ref["k"], case["heads"], case["channels"])
    v_rms, v = sample(cfg, ref["v"], case["heads"], case["channels"])
    # Stored with 17 significant digits; libm may differ in the last bit between machines.
    assert _scaled_err(k, k_rms, case["k"], case["k_rms"]) < 1e-12
    assert _scaled_err(v, v_rms, case["v"], case["v_rms"]) < 1e-12
    np.testing.assert_allclose(k_rms, case["k_rms"], rtol=1e-12)
    np.testing.assert_allclose(v_rms, case["v_rms"], rtol=1e-12)


@pytest.mark.gpu
@pytest.mark.parametrize("case,cfg", CASES, ids=IDS)
def test_cuda_build_matches_stored_values(case, cfg):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34972_gb300.build import build_library
    from tests import gpu_util as gu
    build_library()
    inp = synth.make_inputs(cfg)
    assert input_digest(inp) == case["inputs_sha256"], "the seeded input generator changed"
    k, v, _ = gu.run_build(inp, fill=-3.0)
    toks = np.asarray(case["tokens"])
    _, gk = sample(cfg, gu.gather(k, cfg, toks), case["heads"], case["channels"])
    _, gv = sample(cfg, gu.gather(v, cfg, toks), case["heads"], case["channels"])
    ek = _scaled_err(gk, None, case["k"], case["k_rms"])
    ev = _scaled_err(gv, None, case["v"], case["v_rms"])
    assert ek <= gu.REL_TOL and ev <= gu.REL_TOL, f"{case['name']}: K err {ek:.3e}, V err {ev:.3e}"
