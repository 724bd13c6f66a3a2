"""fq_pack on the GPU is bit-exact with the oracle's packer (layout of framequant.h)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from oracle import pack  # noqa: E402

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.mark.parametrize("n_out,n_in", [(288, 288), (130, 70), (16, 16), (1, 1), (4512, 4512),
                                        (3392, 848), (12112, 4512), (129, 1000)])
def test_pack_bit_exact(n_out, n_in):
    codes = wl.random_codes(5, "gpu-pack", str(n_out), str(n_in), n_out=n_out, n_in=n_in)
    words = torch.full((fq.fq_packed_words(n_out, n_in),), -1, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    fq.fq_pack(torch.from_numpy(codes).to(DEV), n_out, n_in, words, status)
    assert fq.fq_check(status) == 0
    np.testing.assert_array_equal(words.cpu().numpy().view(np.uint32), pack.pack(codes))


def test_pack_flags_out_of_range_codes():
    codes = np.zeros((128, 64), np.uint8)
    codes[5, 7] = 6
    words = torch.zeros(fq.fq_packed_words(128, 64), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    fq.fq_pack(torch.from_numpy(codes).to(DEV), 128, 64, words, status)
    assert fq.fq_check(status) == 7          # FQ_ERR_DEVICE_CHECK
    codes[5, 7] = 2                           # the low two bits of 6 were packed
    np.testing.assert_array_equal(words.cpu().numpy().view(np.uint32), pack.pack(codes))
