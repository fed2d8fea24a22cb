"""The seeded input generators (CPU only)."""
import math

import torch

from paper_2602_07160_gb300 import workloads as W


def test_five_workloads_and_flops():
    assert set(W.WORKLOADS) == {"tiny_f32_causal", "vit_s_full_prior", "lm_causal_d64", "lm_causal_d128",
                                "long_causal_student_t"}
    w = W.WORKLOADS[W.HEADLINE]
    assert (w.B, w.H, w.T, w.d, w.causal) == (4, 16, 8192, 128, True)
    assert w.flops == 4 * 4 * 16 * 8192 * 8192 * 128 / 2
    assert W.WORKLOADS["vit_s_full_prior"].flops == 4 * 64 * 6 * 197 * 197 * 64


def test_shapes_dtypes_and_determinism():
    w = W.WORKLOADS["lm_causal_d64"]
    q, k, v, b = W.make_inputs(w, seed=0, T=100, B=2, H=3)
    assert q.shape == (2, 3, 100, 64) and q.dtype == torch.bfloat16 and q.is_contiguous()
    assert b.shape == (3, 64) and b.dtype == torch.float32
    q2, k2, v2, b2 = W.make_inputs(w, seed=0, T=100, B=2, H=3)
    assert torch.equal(q, q2) and torch.equal(v, v2) and torch.equal(b, b2)
    q3, *_ = W.make_inputs(w, seed=1, T=100, B=2, H=3)
    assert not torch.equal(q, q3)
    assert float(b.min()) >= 0.05 * (1 - 1e-6) and float(b.max()) <= 20.0 * (1 + 1e-6)


def test_tiny_is_fp32():
    q, k, v, b = W.make_inputs(W.WORKLOADS["tiny_f32_causal"])
    assert q.dtype == torch.float32 and q.shape == (1, 1, 64, 16)
    assert float(b.min()) >= 0.1 * (1 - 1e-6) and float(b.max()) <= 10.0 * (1 + 1e-6)


def test_student_t_stress_values():
    w = W.WORKLOADS["long_causal_student_t"]
    q, k, v, b = W.make_inputs(w, T=20000, H=2)
    vf = v.float()
    # channels 0..3 constant over t
    assert torch.all(vf[:, :, :, :4] == vf[:, :, :1, :4])
    # unit variance after the 1/sqrt(3) scaling (t3 has variance 3); heavy tails
    rest = vf[:, :, :, 4:].flatten()
    assert abs(float(rest.var()) - 1.0) < 0.25
    kurt = float(((rest - rest.mean()) ** 4).mean() / rest.var() ** 2)
    assert kurt > 6.0
    assert float(b.min()) >= 1e-3 * (1 - 1e-6) and float(b.max()) <= 100.0 * (1 + 1e-6)
    lb = torch.log(b.double())
    assert float(lb.min()) < math.log(0.01) and float(lb.max()) > math.log(10)


def test_beta_grid():
    g = W.beta_grid(2, 8, [0.0, 1.0, 5.0])
    assert g.shape == (2, 8) and g.dtype == torch.float32
    assert g.flatten().tolist()[:6] == [0.0, 1.0, 5.0, 0.0, 1.0, 5.0]
