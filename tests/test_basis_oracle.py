"""The basis oracle on a synthetic calibration set (CPU only): the
data-driven basis of Section 4.1.2 keeps more energy under top-k pruning than
a random orthogonal basis (the "Random Projection" ablation), for keys,
queries and values."""
import numpy as np

import oracle
from paper_2511_18936_gb300 import synth


def test_data_driven_basis_keeps_more_energy_than_random():
    n_kv, G, n, d, d_model = 2, 2, 512, 128, 256
    Q, K, V, W_O = synth.calibration(n_kv, G, n, d, d_model, seed=0, workload=50, layer=0)
    bo = oracle.basis_oracle
    gen = np.random.default_rng(0)
    for j, (sqk, svo) in enumerate(zip(bo.joint_qk(Q, K, G), bo.joint_vo(V, W_O, G))):
        P_qk, _ = bo.principal_basis(sqk)
        P_vo, _ = bo.principal_basis(svo)
        R = synth.random_orthogonal(d, gen)
        for X, P in ((K[j], P_qk), (Q[j * G], P_qk), (V[j], P_vo)):
            E, Er = bo.energy_curve(X, P), bo.energy_curve(X, R)
            assert abs(E[d] - Er[d]) < 1e-9 * E[d]          # rotations keep the total
            for k in (16, 32, 64):
                assert E[k] > Er[k], (j, k)
            assert E[64] / E[d] > 0.9
