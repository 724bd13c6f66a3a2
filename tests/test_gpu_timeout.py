"""The device-error path of the forward (SURVEY boundary: bounded waits report FQ_ERR_TIMEOUT
through the workspace status word, and the context stays usable), exercised without a GPU
fault: the timeout test hook of fq_forward_opts makes a one-CTA launch wait for a ready stamp
that no call writes, with a short limit (about a millisecond).  The call must end with
FQ_ERR_TIMEOUT and the waiting role recorded; after the workspace is zeroed again, a normal call
on the same workspace and stream must report FQ_OK and match the oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
from fqgpu import DEV, DeviceLayer, activations, assert_parity, oracle_layer, reference  # noqa: E402

pytestmark = pytest.mark.gpu
ROLE_ACTIVATION_PRODUCER = 2      # the role the header's timeout words record for this wait


@pytest.mark.parametrize("M", [8, 40])
def test_injected_wait_times_out_then_the_workspace_recovers(M):
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, torch.bfloat16)
    X = activations("single256", "single", M)
    x = torch.from_numpy(X).to(DEV, torch.bfloat16)
    y = torch.zeros(M, L.d_out, dtype=torch.bfloat16, device=DEV)
    nb = fq.fq_workspace_bytes(M, L.d_in, L.n_in, L.n_out, L.d_out)
    ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)

    fq.fq_linear_forward_ex(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ws, nb,
                            max_sms=1, inject_timeout_cycles=2_000_000)
    assert fq.fq_check(ws) == 6                            # FQ_ERR_TIMEOUT
    words = ws[:32].view(torch.int32).cpu().numpy()
    assert words[4] == ROLE_ACTIVATION_PRODUCER            # who gave up
    assert words[7] % 1000 == 1                            # waiting for the code product's input

    # the context is still usable: zero the workspace, run normally, check against the oracle
    ws.zero_()
    fq.fq_linear_forward_ex(x, M, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ws, nb,
                            max_sms=1)
    assert fq.fq_check(ws) == 0
    assert_parity(y.double().cpu().numpy(), reference(L, X, False), 1e-2)
    assert (ws[16:32].view(torch.int32).cpu().numpy() == 0).all()   # details cleared per call


def test_timeout_details_do_not_outlive_the_workspace_reset():
    """A second workspace used normally after a timed-out one is unaffected (the hook touches
    only the workspace it was given)."""
    L = oracle_layer("single256", "single")
    D = DeviceLayer(L, torch.bfloat16)
    X = activations("single256", "single", 16)
    x = torch.from_numpy(X).to(DEV, torch.bfloat16)
    nb = fq.fq_workspace_bytes(16, L.d_in, L.n_in, L.n_out, L.d_out)
    ws_bad = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    ws_ok = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    y = torch.zeros(16, L.d_out, dtype=torch.bfloat16, device=DEV)
    fq.fq_linear_forward_ex(x, 16, L.d_in, D.T_in, D.C, D.T_out_t, L.d_out, None, y, ws_bad, nb,
                            max_sms=1, inject_timeout_cycles=1_000_000)
    assert fq.fq_check(ws_bad) == 6
    got = D.forward(X, False, ws=ws_ok)
    assert_parity(got, reference(L, X, False), 1e-2)
    np.testing.assert_array_equal(got, D.forward(X, False))
