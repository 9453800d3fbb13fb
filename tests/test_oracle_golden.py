"""The oracle against a layer worked by hand from Lemma 1 (tests/golden)."""
import json
import os

import numpy as np

import oracle

O = oracle.get()
HERE = os.path.dirname(os.path.abspath(__file__))


def test_hand_worked_two_feature_layer():
    with open(os.path.join(HERE, "golden", "lemma1_two_feature_example.json")) as fh:
        g = json.load(fh)
    X = np.array(g["X"])
    W = np.array(g["W"], np.float32).astype(np.float64)
    S = O.sigma(X)
    assert np.array_equal(S, np.array([[2.0, 1.0], [1.0, 2.0]]))
    s, z = O.grid(W, g["bits"])
    assert abs(float(s[0]) - g["scale"]) <= g["tolerance"]["scale_rel"] * g["scale"]
    assert float(z[0]) == g["zero"]
    iters = len(g["codes"])
    r = O.alg1(W, S, s, z, g["bits"], iters, record=True, want_beta=True)
    assert np.array_equal(r["sweep_codes"], np.array(g["codes"], np.uint8))
    assert np.allclose(r["beta"], np.array(g["beta"]), atol=g["tolerance"]["beta_abs"], rtol=0)
    assert np.allclose(r["obj"], g["objective"], rtol=g["tolerance"]["objective_rel"])
