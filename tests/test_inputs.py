"""The seeded synthetic inputs follow the stated recipe: deterministic per
seed, the stated distributions and scales, and the workloads' layer shapes,
block sizes and rates.  CPU only."""
import numpy as np

import oracle
from paper_2111_11581_gb300 import inputs


def _vals(bits, dtype):
    return oracle.to_double(bits, dtype)


def test_generators_are_deterministic_per_seed():
    a = inputs.normal((64, 64), 0.02, inputs.BF16, 5)
    assert np.array_equal(a, inputs.normal((64, 64), 0.02, inputs.BF16, 5))
    assert not np.array_equal(a, inputs.normal((64, 64), 0.02, inputs.BF16, 6))
    u = inputs.uniform((64, 64), -1.0, 1.0, inputs.F16, 5)
    assert np.array_equal(u, inputs.uniform((64, 64), -1.0, 1.0, inputs.F16, 5))


def test_distributions_and_scales():
    n = inputs.normal((512, 512), 0.02, inputs.F16, 11)
    v = _vals(n, inputs.F16)
    assert abs(v.mean()) < 1e-3 and abs(v.std() - 0.02) < 5e-4
    u = _vals(inputs.uniform((512, 512), -1.0, 1.0, inputs.BF16, 12), inputs.BF16)
    assert u.min() >= -1.0 and u.max() <= 1.0
    assert abs(u.mean()) < 1e-2 and abs(u.var() - 1.0 / 3.0) < 1e-2
    b = inputs.bias(100000, 0.01, 13)
    assert b.dtype == np.float32 and abs(b.std() - 0.01) < 2e-4
    assert abs(inputs.kaiming_std(1152) - (2.0 / 1152) ** 0.5) < 1e-15


def test_workload_layers():
    fc = inputs.fc512()
    assert (fc.M, fc.K, fc.N, fc.bm, fc.bk, fc.rate) == (512, 512, 64, 16, 16, 4.0)
    cv = inputs.conv3x3_128()
    assert (cv.M, cv.C, cv.kh, cv.N, cv.H, cv.pad, cv.bm, cv.bk, cv.rate) == \
        (128, 128, 3, 128, 16, 1, 8, 4, 3.0)
    w = _vals(inputs.layer_weight(cv, inputs.F16), inputs.F16)
    assert abs(w.std() - inputs.kaiming_std(128 * 9)) < 0.02 * inputs.kaiming_std(128 * 9)
    vgg = inputs.vgg16_cifar()
    convs = [l for l in vgg if l.kind == "conv"]
    assert len(convs) == 13 and convs[0].scheme < 0
    assert all(l.bm == 8 and l.bk == 4 and l.rate == 8.0 for l in convs[1:])
    assert vgg[-1].kind == "fc" and (vgg[-1].M, vgg[-1].K, vgg[-1].N) == (10, 512, 256)
    rn = inputs.resnet50_imagenet()
    pruned = [l for l in rn if l.scheme >= 0]
    assert len(pruned) == 53 and rn[0].scheme < 0
    assert abs(np.mean([l.rate for l in pruned]) - 6.0) < 1e-9
    for l in pruned:
        if l.kind == "conv" and l.kh == 3:
            assert (l.bm, l.bk, l.rate) == (16, 8, 8.0)
        else:
            assert (l.bm, l.bk) == (32, 32)
    for M, K, N in inputs.GEMM_SHAPES:
        g = inputs.gemm_point(M, K, N, 128, 32, 4.0, inputs.BF16)
        x = _vals(inputs.layer_input(g, inputs.BF16)[:64], inputs.BF16)
        assert g.N == N and x.min() >= -1.0 and x.max() <= 1.0
