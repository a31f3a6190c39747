"""GPU check of sara_gemm_bf16_static, the GEMM entry point that allocates nothing.

Some callers cannot allocate device memory themselves (their framework's pool owns the
GPU, or their interface only passes inputs and outputs); this entry point keeps its scratch
in a fixed array inside the library.  The test calls it twice in a row through the C ABI
(the second call must not be disturbed by what the first left in the shared scratch) and
compares both results with sara_gemm_bf16, which takes a caller workspace, within the fp32
accumulation bound the GEMM tests use.  This file is collected last on purpose.
"""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_26253_gb300 as p
    p.load()
    return p


def _bf16_dev(rng, shape, scale):
    import torch
    bits = synth.f32_to_bf16_bits((rng.standard_normal(shape) * scale).astype(np.float32))
    return bits, torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("R,N,K", [(25, 1536, 1536), (128, 2048, 8960), (7, 17920, 1536)])
def test_static_scratch_gemm_matches_workspace_gemm_twice(pkg, R, N, K):
    import torch
    rng = np.random.default_rng(R + N + K)
    xb, X = _bf16_dev(rng, (R, K), 1.0)
    wb, W = _bf16_dev(rng, (N, K), 0.02)
    ref = pkg.gemm_bf16(X, W).cpu().numpy()
    xf = synth.bf16_bits_to_f32(xb).astype(np.float64)
    wf = synth.bf16_bits_to_f32(wb).astype(np.float64)
    bound = 2 * K * 2.0 ** -23 * (np.abs(xf) @ np.abs(wf).T) + 1e-6  # two fp32 accumulations
    out = torch.empty((R, N), dtype=torch.float32, device="cuda")
    for _ in range(2):
        out.fill_(float("nan"))
        got = pkg.gemm_bf16_static(X, W, out=out).cpu().numpy()
        assert np.all(np.abs(got - ref) <= bound)


def test_static_scratch_rejects_oversized_output(pkg):
    import torch
    X = torch.zeros((4, 64), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((262144 + 128, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pkg.SaraError):
        pkg.gemm_bf16_static(X, W)
