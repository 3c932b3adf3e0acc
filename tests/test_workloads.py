"""The seeded synthetic inputs (CPU): G_{i,t} = S + c Xi_{i,t} / sqrt(n) with S = U_b diag(s) V_b^T.

Checks that the generator produces what the input recipe states: the configurations' shapes and
sizes, a fixed low-rank part with exactly the configured singular values, noise of the configured
scale that is fresh per node and step and reproducible per seed, round-to-nearest-even bf16
rounding, and the device (torch) generator following the same recipe.
"""
import math

import numpy as np
import pytest

import workloads as W


def test_configuration_sizes():
    cfg2 = W.config("cfg2_resnet")
    assert cfg2.shapes == ((64, 576), (64, 576), (128, 1152), (128, 1152), (256, 2304), (256, 2304),
                           (512, 4608), (512, 4608))
    assert (cfg2.N, cfg2.r, cfg2.basis_rank, cfg2.tau, cfg2.grad_dtype) == (8, 8, 16, 50, "f32")
    assert cfg2.matrix_elems() == 6_266_880
    assert W.config("cfg1_tiny").shapes == ((256, 128),)
    assert W.config("cfg3_llama_d2048").matrix_elems() == 616_562_688
    assert len(W.config("cfg3_llama_d2048").shapes) == 84
    assert W.config("cfg4_refresh").shapes == ((4096, 11008),)
    assert W.config("cfg5_llama_d4096").matrix_elems() == 1_619_001_344
    assert len(W.config("cfg5_llama_d4096").shapes) == 56


@pytest.mark.parametrize("name", ["cfg1_tiny", "cfg2_resnet"])
def test_low_rank_part_has_the_configured_spectrum(name):
    cfg = W.config(name)
    prob = W.make_problem(cfg)
    for li, (m, n) in enumerate(cfg.shapes[:3]):
        rho = min(cfg.rho, m, n)
        Ub, Vb = prob.Ub[li], prob.Vb[li]
        np.testing.assert_allclose(Ub.T @ Ub, np.eye(rho), atol=1e-12)
        np.testing.assert_allclose(Vb.T @ Vb, np.eye(rho), atol=1e-12)
        sv = np.linalg.svd(prob.S(li), compute_uv=False)
        want = np.array([cfg.spectrum(k) for k in range(1, rho + 1)])
        np.testing.assert_allclose(sv[:rho], want, rtol=1e-10)
        assert np.all(sv[rho:] < 1e-12 * sv[0])


def test_noise_scale_freshness_and_seeding():
    cfg = W.config("cfg2_resnet")
    prob = W.make_problem(cfg)
    li = 4                                               # 256 x 2304
    m, n = cfg.shapes[li]
    G0 = W.gradients_numpy(prob, li, 0, workers=[0, 1])
    G1 = W.gradients_numpy(prob, li, 1, workers=[0])
    S = prob.S(li)
    xi = (G0 - S) * math.sqrt(n) / cfg.noise             # should be N(0, 1) up to fp32 rounding
    assert abs(xi.mean()) < 0.01
    assert abs(xi.std() - 1.0) < 0.01
    # fresh per node and per step (correlations of independent N(0,1) fields ~ 1/sqrt(m n))
    c_nodes = np.corrcoef(xi[0].ravel(), xi[1].ravel())[0, 1]
    c_steps = np.corrcoef(xi[0].ravel(), ((G1[0] - S) * math.sqrt(n) / cfg.noise).ravel())[0, 1]
    assert abs(c_nodes) < 0.01 and abs(c_steps) < 0.01
    # reproducible from the seed, node by node
    np.testing.assert_array_equal(W.gradients_numpy(prob, li, 0, workers=[1])[0], G0[1])
    other = W.make_problem(cfg, seed=cfg.master_seed + 1)
    assert not np.allclose(other.S(li), S)


def test_bf16_rounding_is_round_to_nearest_even():
    one = 1.0
    ulp = 2.0 ** -7                                      # bf16 spacing in [1, 2)
    x = np.array([one, one + ulp / 2, one + 1.5 * ulp, one + 0.75 * ulp, -(one + ulp / 2), 3.0e38])
    y = W.round_to_dtype_numpy(x, "bf16")
    np.testing.assert_array_equal(y[:5], [one, one, one + 2 * ulp, one + ulp, -one])   # ties to even
    bits = y.astype(np.float32).view(np.uint32)
    assert np.all((bits & 0xFFFF) == 0)                  # representable in bf16
    f32 = W.round_to_dtype_numpy(np.array([0.1]), "f32")
    assert f32[0] == float(np.float32(0.1))


def test_device_generator_follows_the_recipe():
    torch = pytest.importorskip("torch")
    cfg = W.config("cfg2_resnet")
    prob = W.make_problem(cfg)
    li = 2                                               # 128 x 1152
    m, n = cfg.shapes[li]
    G = W.gradients_torch(prob, li, 0, device="cpu", workers=[0, 1])
    assert len(G) == 2 and G[0].shape == (m, n) and G[0].dtype == torch.float32
    S = prob.S(li)
    xi = [(g.double().numpy() - S) * math.sqrt(n) / cfg.noise for g in G]
    for x in xi:
        assert abs(x.mean()) < 0.02 and abs(x.std() - 1.0) < 0.02
    assert abs(np.corrcoef(xi[0].ravel(), xi[1].ravel())[0, 1]) < 0.02
    G_again = W.gradients_torch(prob, li, 0, device="cpu", workers=[1])
    assert torch.equal(G_again[0], G[1])
