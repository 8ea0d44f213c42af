"""NABF on the GPU (af1_nabf_factorize) against the FP64 oracle
(oracle/af1_nabf_oracle.py) and the invariants of its output."""
import numpy as np
import pytest
import torch

import synth
from oracle import af1_nabf_oracle as N
from oracle import af1_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


def _weights(seed, m, n, rank=None, noise=0.01):
    """Synthetic weights: Gaussian, or a rank-`rank` matrix plus noise."""
    g = synth.rng(seed)
    if rank is None:
        return g.normal(0.0, 0.02, size=(m, n))
    return g.normal(size=(m, rank)) @ g.normal(size=(rank, n)) * 0.01 + g.normal(0.0, noise, size=(m, n))


def _recon(U, V, a, s, b):
    return (a[:, None] * (U.astype(np.float64) * s[None, :])) @ V.astype(np.float64).T * b[None, :]


@pytest.mark.parametrize("m,n,r", [(48, 40, 8), (96, 128, 24), (130, 70, 33)])
@pytest.mark.parametrize("iters", [0, 1, 3])
@pytest.mark.parametrize("compensate", [True, False])
def test_nabf_matches_oracle(P, m, n, r, iters, compensate):
    """FP32 on the GPU against FP64, on nearly rank-deficient weights (so the
    null-space projectors keep 1-5 vectors) whose Gram matrices stay well
    conditioned (kappa(A0^T A0 + rho I) <= 1e3). With noise 0.002 instead of
    0.01 (kappa 1.2e4 at 130 x 70, r = 33) the FP32 solves already move 10 %
    of the initial signs of B: the GPU path computes in FP32."""
    W = _weights(m + n + iters, m, n, rank=r // 2 + 1)
    g = synth.rng(7)
    i_s, o_s = g.uniform(0.5, 2.0, n), g.uniform(0.5, 2.0, m)
    ref = N.nabf(W, r, iters, rho=1e-2, eta=0.01, eps=1e-8, power_iters=30, seed=11, in_scale=i_s, out_scale=o_s,
                 compensate=compensate)
    t = lambda v: torch.tensor(v, dtype=torch.float32, device="cuda")
    out = P.nabf_factorize(t(W), r, iters=iters, rho=1e-2, eta=0.01, eps=1e-8, power_iters=30, seed=11,
                           in_scale=t(i_s), out_scale=t(o_s), compensate=compensate)
    U, V = out["U"].cpu().numpy(), out["V"].cpu().numpy()
    agree = min((U == ref["U"]).mean(), (V == ref["V"]).mean())
    assert agree >= 0.999, agree
    Wg = _recon(U, V, *(out[k].double().cpu().numpy() for k in ("a", "s", "b")))
    Wr = _recon(ref["U"], ref["V"], ref["a"], ref["s"], ref["b"])
    assert np.linalg.norm(Wg - Wr) / np.linalg.norm(Wr) <= 2e-3
    np.testing.assert_allclose(out["objective"], ref["objective"], rtol=2e-3, atol=1e-6)
    assert out["q_left"] == list(ref["q_left"]) and out["q_right"] == list(ref["q_right"])


def test_nabf_history_matches_its_output(P):
    """The last objective is the error of the returned AF1 layer on W'."""
    m, n, r = 1024, 768, 256
    W = _weights(3, m, n, rank=64)
    g = synth.rng(4)
    i_s, o_s = g.uniform(0.5, 2.0, n), g.uniform(0.5, 2.0, m)
    t = lambda v: torch.tensor(v, dtype=torch.float32, device="cuda")
    out = P.nabf_factorize(t(W), r, iters=6, rho=1e-4, in_scale=t(i_s), out_scale=t(o_s))
    Wh = _recon(out["U"].cpu().numpy(), out["V"].cpu().numpy(), *(out[k].double().cpu().numpy() for k in ("a", "s", "b")))
    Wp = o_s[:, None] * W * i_s[None, :]
    err = np.linalg.norm(Wp - o_s[:, None] * Wh * i_s[None, :]) ** 2 / np.linalg.norm(Wp) ** 2
    assert err == pytest.approx(out["objective"][-1], rel=1e-3)
    assert out["objective"][-1] < out["objective"][0]
    assert all(0 <= q <= r for q in out["q_left"] + out["q_right"])
    assert set(np.unique(out["U"].cpu().numpy())) <= {-1, 1}


def test_nabf_layer_runs_through_the_forward_pass(P):
    """Quantize with NABF, pack at FP16 scales, run the decode path: the
    output equals the oracle's forward of the same packed layer."""
    m, n = 512, 384
    r = O.rank_for_budget(m, n, 1)
    W = _weights(9, m, n, rank=48)
    out = P.nabf_factorize(torch.tensor(W, dtype=torch.float32, device="cuda"), r, iters=4, rho=1e-4)
    a16, s16, b16 = (out[k].half() for k in ("a", "s", "b"))
    layer = P.Layer.from_signs(out["U"], out["V"], a16, s16, b16)
    x = synth.activations_f16(synth.rng(1), 3, n)
    y = layer.forward(torch.from_numpy(x.view(np.float16)).cuda().reshape(3, n), out_dtype=torch.float32)
    torch.cuda.synchronize()
    bits = lambda tns: tns.cpu().numpy().view(np.uint16)
    ref = O.forward_from_packed(O.pack_U(out["U"].cpu().numpy()), O.pack_V(out["V"].cpu().numpy()), bits(a16),
                                bits(s16), bits(b16), x, m, n, r)
    assert O.rowwise_rel_err(y.double().cpu().numpy(), ref) <= 2e-3
    layer.free()
