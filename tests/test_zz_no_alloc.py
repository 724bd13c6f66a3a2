"""fq_linear_forward_static: the forward for callers that cannot allocate device memory (a
host framework that owns all allocations, a plugin interface without a workspace argument, a
C program without an allocator) uses a scratch array inside the library instead of a
caller-provided workspace.  Its output must match fq_linear_forward's, call after call, and
sizes beyond the array are refused.  This file is collected last on purpose."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
from fqgpu import DEV, DeviceLayer, activations, oracle_layer, assert_parity, rel_frobenius  # noqa: E402

pytestmark = pytest.mark.gpu
TOL = {torch.bfloat16: 1e-2, torch.float32: 1e-5}


@pytest.mark.parametrize("dtype,M", [(torch.bfloat16, 16), (torch.bfloat16, 40),
                                     (torch.float32, 16), (torch.float32, 40),
                                     (torch.bfloat16, 128), (torch.bfloat16, 300)],
                         ids=["bf16-16", "bf16-40", "fp32-16", "fp32-40", "bf16-128",
                              "bf16-300"])
def test_static_matches_workspace_forward_twice(dtype, M):
    """M <= 64 runs the fused decode kernel through the array, M = 128 and 300 the tensor-core
    kernels (whose split-K counters must be left zeroed for the next call)."""
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, dtype)
    mode = fq.FQ_BF16 if dtype == torch.bfloat16 else fq.FQ_FP32_DEBUG
    X = activations("single256", "single", M)
    ref = D.forward(X, True)                       # the existing entry point, own workspace
    x = torch.from_numpy(X).to(DEV, dtype)
    for _ in range(2):                             # two calls in a row share the array
        y = torch.full((M, L.d_out), float("nan"), dtype=dtype, device=DEV)
        fq.fq_linear_forward_static(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, D.gamma, y,
                                    mode)
        torch.cuda.synchronize()
        assert fq.fq_static_check() == 0
        got = y.double().cpu().numpy()
        assert np.isfinite(got).all()
        assert_parity(got, ref, TOL[dtype])


def test_static_refuses_sizes_beyond_the_array():
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, torch.bfloat16)
    # a token count whose intermediates exceed FQ_STATIC_SCRATCH_BYTES
    M = fq.FQ_STATIC_SCRATCH_BYTES // (2 * (L.n_in + L.n_out)) + 64
    assert fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out) > fq.FQ_STATIC_SCRATCH_BYTES
    x = torch.zeros(M, L.d_in, dtype=torch.bfloat16, device=DEV)
    y = torch.full((M, L.d_out), 3.0, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(fq.FrameQuantError) as e:
        fq.fq_linear_forward_static(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y)
    assert e.value.status == 3                     # FQ_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert (y == 3.0).all()
