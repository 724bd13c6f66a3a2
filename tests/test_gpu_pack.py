"""fq_pack on the GPU is bit-exact with the oracle's packer (layout of framequant.h), fills the
descriptor the forward takes (the per-row scale and zero with the codes, Appendix K), and
flags out-of-range codes and non-finite scales or zeros."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_06082_gb300 as fq  # noqa: E402
import workloads as wl  # noqa: E402
from oracle import pack, quant  # noqa: E402

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _scale_zero(n_out, seed=0):
    sc, ze = wl.random_scale_zero(seed, "gpu-pack-sz", n_out=n_out, mag=0.01)
    return (torch.from_numpy(sc.view(np.int16).copy()).to(DEV),
            torch.from_numpy(ze.view(np.int16).copy()).to(DEV), sc, ze)


@pytest.mark.parametrize("n_out,n_in", [(288, 288), (130, 70), (16, 16), (1, 1), (4512, 4512),
                                        (3392, 848), (12112, 4512), (129, 1000)])
def test_pack_bit_exact(n_out, n_in):
    codes = wl.random_codes(5, "gpu-pack", str(n_out), str(n_in), n_out=n_out, n_in=n_in)
    words = torch.full((fq.fq_packed_words(n_out, n_in),), -1, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    s, z, sc, ze = _scale_zero(n_out)
    C = fq.fq_pack(torch.from_numpy(codes).to(DEV), s, z, n_out, n_in, words, status)
    assert fq.fq_check(status) == 0
    np.testing.assert_array_equal(words.cpu().numpy().view(np.uint32), pack.pack(codes))
    # the descriptor: sizes, row pitch, width, and the scale and zero it carries
    assert (C.n_out, C.n_in, C.bits) == (n_out, n_in, 2)
    assert C.ld_words == 4 * (-(-n_in // 64))
    assert C.ld_words * pack.padded(n_out, n_in)[0] == words.numel()
    assert C.scale.data_ptr() == s.data_ptr() and C.zero.data_ptr() == z.data_ptr()
    np.testing.assert_array_equal(C.scale.cpu().numpy().view(np.float16), sc)
    np.testing.assert_array_equal(C.zero.cpu().numpy().view(np.float16), ze)


def test_pack_carries_the_oracle_rtn_scale_and_zero():
    """Codes, scale and zero of the oracle's RTN of a coefficient matrix go in as one unit; the
    packed words and the fp16 bit patterns come back unchanged."""
    C_f = wl.rng(11, "gpu-pack-rtn").standard_normal((256, 320)) * 0.02
    q, sc, ze = quant.rtn(C_f)
    words = torch.zeros(fq.fq_packed_words(256, 320), dtype=torch.int32, device=DEV)
    s = torch.from_numpy(sc.view(np.int16).copy()).to(DEV)
    z = torch.from_numpy(ze.view(np.int16).copy()).to(DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    P = fq.fq_pack(torch.from_numpy(q).to(DEV), s, z, 256, 320, words, status)
    assert fq.fq_check(status) == 0
    np.testing.assert_array_equal(words.cpu().numpy().view(np.uint32), pack.pack(q))
    assert P.scale.cpu().numpy().view(np.uint16).tobytes() == sc.view(np.uint16).tobytes()
    assert P.zero.cpu().numpy().view(np.uint16).tobytes() == ze.view(np.uint16).tobytes()


def test_pack_flags_out_of_range_codes():
    codes = np.zeros((128, 64), np.uint8)
    codes[5, 7] = 6
    words = torch.zeros(fq.fq_packed_words(128, 64), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    s, z, _, _ = _scale_zero(128)
    fq.fq_pack(torch.from_numpy(codes).to(DEV), s, z, 128, 64, words, status)
    assert fq.fq_check(status) == 7          # FQ_ERR_DEVICE_CHECK
    codes[5, 7] = 2                           # the low two bits of 6 were packed
    np.testing.assert_array_equal(words.cpu().numpy().view(np.uint32), pack.pack(codes))


@pytest.mark.parametrize("which,bits", [("scale", 0x7C00), ("zero", 0xFC00), ("scale", 0x7E00)])
def test_pack_flags_non_finite_scale_or_zero(which, bits):
    codes = np.zeros((128, 64), np.uint8)
    words = torch.zeros(fq.fq_packed_words(128, 64), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    s, z, _, _ = _scale_zero(128)
    t = s if which == "scale" else z
    t[77] = np.uint16(bits).view(np.int16).item()      # +inf, -inf, NaN
    fq.fq_pack(torch.from_numpy(codes).to(DEV), s, z, 128, 64, words, status)
    assert fq.fq_check(status) == 7
