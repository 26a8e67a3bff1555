"""The seeded input generator: determinism, shapes and the stated statistics."""

import numpy as np
import torch

import workload as wl


def test_deterministic_and_shaped():
    spec = wl.VideoSpec(T=6, H=5, W=7, D=16, Lq=3, cuts=1, seed=77)
    X1, Q1, m1 = wl.make_video(spec)
    X2, Q2, m2 = wl.make_video(spec)
    assert X1.shape == (6, 5, 7, 16) and Q1.shape == (3, 16) and X1.dtype == torch.bfloat16
    assert torch.equal(X1, X2) and torch.equal(Q1, Q2) and m1 == m2
    assert len(m1["cuts"]) == 1 and 1 <= m1["cuts"][0] <= 5


def test_field_statistics():
    spec = wl.VideoSpec(T=40, H=12, W=12, D=64, dtype="f32", Lq=4, ar=0.9, cuts=0, seed=5)
    X, Q, _ = wl.make_video(spec)
    x = X.double().numpy()
    assert abs(x.std() - np.sqrt(1.0 + 0.01)) < 0.08             # unit field + 0.1 noise
    lag1 = np.mean(x[1:] * x[:-1]) / np.mean(x * x)
    assert abs(lag1 - 0.9 / 1.01) < 0.06                          # AR(1) in time
    sp = np.mean(x[:, 1:] * x[:, :-1]) / np.mean(x * x)
    assert sp > 0.8                                               # smooth in space
    assert abs(Q.double().std().item() - 1 / 8.0) < 0.03          # std 1/sqrt(D)


def test_smoothing_rows_unit_norm():
    K = wl.smoothing_matrix(13, 3.0)
    assert np.allclose(np.linalg.norm(K, axis=1), 1.0)


def test_configs_and_batch():
    assert set(wl.CONFIGS) == {"tiny_f32_16x14x14", "video64_13x13_bf16",
                               "video128_16x16_objects", "video256_27x27_bf16"}
    specs = wl.batch_specs()
    assert len(specs) == 32 and all(8 <= s.Lq <= 128 for s in specs)
    assert set(s.ratio for s in specs) <= {0.05, 0.1, 0.25}
    assert [s.seed for s in specs] == list(range(2000, 2032))
