"""The C-ABI library loads, exports every entry point include/framequant.h declares, and
rejects bad arguments on the host with a status and without touching the GPU."""
import ctypes
import os
import re

import pytest

import paper_2403_06082_gb300 as fq

INCLUDE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")


def _declared():
    names = set()
    for f in sorted(os.listdir(INCLUDE)):
        if f.endswith(".h"):
            text = re.sub(r"/\*.*?\*/", "", open(os.path.join(INCLUDE, f)).read(), flags=re.S)
            names |= set(re.findall(r"\b(fq_[a-z_]+)\s*\(", text))
    return sorted(names)


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(fq.lib_path()):
        import __graft_entry__
        __graft_entry__.build()
    return fq.lib()


def test_exports_every_declared_symbol(L):
    names = _declared()
    assert set(names) == set(fq.EXPORTED)
    for n in names:
        assert hasattr(L, n), n


def test_packed_words(L):
    assert fq.fq_packed_words(288, 288) == 384 * 320 // 16
    assert fq.fq_packed_words(128, 64) == 512
    assert fq.fq_packed_words(0, 64) == 0
    assert fq.fq_packed_words(12112, 4512) == 12160 * 4544 // 16


def test_status_strings(L):
    for k, v in fq.STATUS.items():
        assert fq.fq_status_str(k) == v


def test_workspace_bytes(L):
    a = fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, fq.FQ_BF16)
    b = fq.fq_workspace_bytes(2048, 4096, 4512, 4512, 4096, fq.FQ_BF16)
    assert 0 < a < b
    assert fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, fq.FQ_FP32_DEBUG) > 0
    assert fq.fq_workspace_bytes(0, 4096, 4512, 4512, 4096, fq.FQ_BF16) == 0
    assert fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, 7) == 0
    # z and u alone are M * (n_in + n_out) bf16
    assert b >= 2048 * (4512 + 4512) * 2


def _P(words, scale, zero, n_out, n_in, ld=None, bits=2):
    """A packed descriptor as fq_pack fills it (ld_words = 4 ceil(n_in / 64), bits = 2)."""
    return fq._Packed(words, scale, zero, n_out, n_in, fq.ld_words(n_in) if ld is None else ld,
                      bits)


def _call(L, x=0x1000, M=8, d_in=256, T_in=0x2000, C=None, T_out=0x3000, d_out=256, gamma=None,
          y=0x4000, ws=0x10000, ws_bytes=1 << 30, mode=0):
    C = C or _P(0x5000, 0x6000, 0x7000, 288, 288)
    return L.fq_linear_forward(x, M, d_in, T_in, ctypes.byref(C), T_out, d_out, gamma, y, ws,
                               ws_bytes, mode, None)


def test_host_validation_without_gpu(L):
    # every rejection happens before any device work (the pointers here are never touched)
    assert _call(L, x=None) == 1
    assert _call(L, y=None) == 1
    assert _call(L, M=0) == 1
    assert _call(L, d_in=-8) == 1
    assert _call(L, mode=5) == 1
    assert _call(L, C=_P(0, 0x6000, 0x7000, 288, 288)) == 1
    assert _call(L, C=_P(0x5000, 0x6000, 0x7000, 0, 288)) == 1
    assert _call(L, x=0x1002) == 2                      # misaligned pointer
    assert _call(L, d_in=260) == 2                      # row pitch not 16 bytes
    assert _call(L, C=_P(0x5000, 0x6000, 0x7000, 280, 288)) == 2   # n_out not a multiple of 16
    assert _call(L, ws=None) == 4
    assert _call(L, ws_bytes=1024) == 4
    assert _call(L, ws=0x10010) == 2                    # workspace not 256-byte aligned
    assert _call(L, C=_P(0x5000, 0x6000, 0x7000, 288, 288, ld=16)) == 1   # wrong row pitch
    assert _call(L, C=_P(0x5000, 0x6000, 0x7000, 288, 288, bits=3)) == 3  # only 2-bit codes
    assert _call(L, C=_P(0x5000, 0x6008, 0x7000, 288, 288)) == 2          # scale misaligned


def test_pack_host_validation_without_gpu(L):
    def pack(codes=0x1000, scale=0x2000, zero=0x3000, n_out=128, n_in=64, words=0x4000,
             out=True):
        o = fq._Packed()
        o.words = words
        st = L.fq_pack(codes, scale, zero, n_out, n_in, ctypes.byref(o) if out else None, None,
                       None)
        return st, o
    assert pack(codes=None)[0] == 1
    assert pack(scale=None)[0] == 1
    assert pack(zero=None)[0] == 1
    assert pack(words=None)[0] == 1
    assert pack(out=False)[0] == 1
    assert pack(n_in=0)[0] == 1
    assert pack(words=0x4004)[0] == 2
    assert pack(scale=0x2002)[0] == 2
    st, o = pack(zero=0x3008)
    assert st == 2 and o.n_out == 0 and o.bits == 0          # a refused call leaves *out alone


def test_valid_bf16_request_needs_sm103(L):
    try:
        import torch
        if torch.cuda.is_available():
            pytest.skip("a GPU is present")
    except ImportError:
        pass
    # no CUDA device: the bf16 path refuses instead of falling back to anything
    assert _call(L) == 3


def _frame(k=18, rho=16, d=256, tiles=0x8000):
    return fq._Frame(k, rho, d, 0, 0, None, None, None, None, None, None, None, tiles, 0x9000, 6,
                     tiles, 0xA000, 6)


def _call_implicit(L, x=0x1000, M=8, Fi=None, C=None, Fo=None, gamma=None, y=0x4000,
                   ws=0x10000, ws_bytes=1 << 30, max_sms=0):
    C = C or _P(0x5000, 0x6000, 0x7000, 288, 288)
    Fi, Fo = Fi or _frame(), Fo or _frame()
    return L.fq_linear_forward_implicit(x, M, ctypes.byref(Fi), ctypes.byref(C), ctypes.byref(Fo),
                                        gamma, y, ws, ws_bytes, max_sms, None)


def test_implicit_frame_sizes_and_validation(L):
    # (k, rho, d) needs rho even, d a multiple of rho and k >= d / rho (tight modulation)
    assert fq.fq_frame_implicit_bytes(18, 16, 256, 16, 16) > 0
    assert fq.fq_frame_implicit_bytes(282, 16, 4096, 64, 64) > 0
    assert fq.fq_frame_implicit_bytes(18, 16, 256, 0, 0) < fq.fq_frame_implicit_bytes(18, 16, 256, 16, 16)
    assert fq.fq_frame_implicit_bytes(15, 16, 256, 16, 16) == 0     # k < w = 16
    assert fq.fq_frame_implicit_bytes(18, 15, 255, 15, 17) == 0     # rho odd
    assert fq.fq_frame_implicit_bytes(18, 16, 264, 8, 33) == 0      # d not a multiple of rho
    assert fq.fq_frame_implicit_bytes(18, 16, 256, 16, 8) == 0      # a * b != d
    assert fq.fq_implicit_workspace_bytes(16, 4096, 4512, 4512, 4096) > \
        fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, fq.FQ_BF16)
    assert fq.fq_implicit_workspace_bytes(65, 4096, 4512, 4512, 4096) == 0
    out = fq._Frame()
    assert L.fq_frame_implicit(15, 16, 256, None, 0x1000, 1 << 20, ctypes.byref(out), None) == 1
    assert L.fq_frame_implicit(18, 16, 256, None, None, 1 << 20, ctypes.byref(out), None) == 4
    assert L.fq_frame_implicit(18, 16, 256, None, 0x1010, 1 << 20, ctypes.byref(out), None) == 2


def test_implicit_host_validation_without_gpu(L):
    assert _call_implicit(L, x=None) == 1
    assert _call_implicit(L, M=0) == 1
    assert _call_implicit(L, max_sms=-1) == 1
    assert _call_implicit(L, Fi=_frame(k=15)) == 1                  # not a tight frame
    assert _call_implicit(L, Fi=_frame(tiles=None)) == 1
    assert _call_implicit(L, C=_P(0x5000, 0x6000, 0x7000, 288, 304)) == 1   # n_in != k rho
    assert _call_implicit(L, x=0x1002) == 2
    assert _call_implicit(L, ws=None) == 4
    assert _call_implicit(L, ws=0x10010) == 2
    assert _call_implicit(L, M=65) == 3                             # decode batches only
    assert _call_implicit(L, ws_bytes=1024) == 4


def test_forward_ex_host_validation_without_gpu(L):
    def ex(opts, **kw):
        C = _P(0x5000, 0x6000, 0x7000, 288, 288)
        a = dict(x=0x1000, M=8, d_in=256, T_in=0x2000, T_out=0x3000, d_out=256, y=0x4000)
        a.update(kw)
        return L.fq_linear_forward_ex(a["x"], a["M"], a["d_in"], a["T_in"], ctypes.byref(C),
                                      a["T_out"], a["d_out"], None, a["y"], 0x10000, 1 << 30, 0,
                                      ctypes.byref(opts) if opts is not None else None, None)
    assert ex(fq._Opts(-1, None, 0)) == 1                  # negative SM budget
    assert ex(fq._Opts(0, None, 4096)) == 1                # range without a pointer
    assert ex(fq._Opts(0, 0x9008, 4096)) == 2              # range start not 16-byte aligned
    assert ex(fq._Opts(0, 0x9000, 4096), x=None) == 1
    # the timeout test hook: one-CTA decode launches only, never negative
    assert ex(fq._Opts(0, None, 0, 100000)) == 1           # needs max_sms = 1
    assert ex(fq._Opts(1, None, 0, -5)) == 1
    assert ex(fq._Opts(1, None, 0, 100000), M=100) == 1    # not the M <= 64 kernel


def test_rotation_validation_without_gpu(L):
    """A rotation whose perm is not a permutation, or whose signs are not +-1, is refused on
    the host by both frame builders."""
    import numpy as np
    a = b = 16
    ga = np.eye(a)
    gb = np.eye(b)

    def rot(perm, signs):
        keep = [np.ascontiguousarray(ga), np.ascontiguousarray(gb),
                np.ascontiguousarray(perm, np.int64), np.ascontiguousarray(signs, np.float64)]
        return fq._Rotation(a, b, *(k.ctypes.data for k in keep)), keep

    good_perm, good_signs = np.arange(256), np.ones(256)
    dup = good_perm.copy()
    dup[3] = 4
    half = good_signs.copy()
    half[7] = 0.5
    out = fq._Frame()
    for perm, signs in ((dup, good_signs), (good_perm, half)):
        r, keep = rot(perm, signs)
        assert L.fq_frame_build(18, 16, 256, ctypes.byref(r), 0x1000, 0x2000, 1 << 30, None) == 1
        assert L.fq_frame_implicit(18, 16, 256, ctypes.byref(r), 0x1000, 1 << 30,
                                   ctypes.byref(out), None) == 1
        del keep


def test_dense_path_sizes_and_validation_without_gpu(L):
    assert fq.fq_dense_workspace_bytes(0, 256, 256) == 0
    assert fq.fq_dense_workspace_bytes(2048, 4096, 4096) > 0
    assert fq.fq_reconstruct_workspace_bytes(4096, 4512, 4512, 4096) >= 4096 * 4096 * 2 * 2
    assert fq.fq_reconstruct_workspace_bytes(0, 4512, 4512, 4096) == 0
    C = _P(0x5000, 0x6000, 0x7000, 288, 288)
    assert L.fq_reconstruct_weight(None, ctypes.byref(C), 0x3000, 256, 256, None, 0x4000,
                                   0x10000, 1 << 30, None) == 1
    assert L.fq_reconstruct_weight(0x2000, ctypes.byref(C), 0x3000, 256, 256, None, 0x4002,
                                   0x10000, 1 << 30, None) == 2
    assert L.fq_reconstruct_weight(0x2000, ctypes.byref(C), 0x3000, 256, 256, None, 0x4000,
                                   0x10000, 1024, None) == 4
    assert L.fq_dense_forward(None, 8, 256, 0x2000, 256, 0x4000, 0x10000, 1 << 30, None) == 1
    assert L.fq_dense_forward(0x1000, 8, 260, 0x2000, 256, 0x4000, 0x10000, 1 << 30, None) == 2
    assert L.fq_dense_forward(0x1000, 8, 256, 0x2000, 256, 0x4000, 0x10000, 64, None) == 4


def test_group_sizes_and_validation_without_gpu(L):
    C = _P(0x5000, 0x6000, 0x7000, 4512, 4512)
    Cg = _P(0x5000, 0x6000, 0x7000, 12112, 4512)

    def layer(x=0x1000, y=0x4000, C=C, d_out=4096, ti=None, to=None):
        return fq._Layer(x, 4096, 0x2000, ctypes.pointer(C), 0x3000, d_out, None, y, ti, to)

    def arr(*ls):
        a = (fq._Layer * len(ls))()
        for i, l_ in enumerate(ls):
            a[i] = l_
        return a
    one = fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096)
    g3 = L.fq_group_workspace_bytes(16, 3, arr(layer(), layer(y=0x8000), layer(y=0x9000)))
    # the header once, then z and u of every layer
    assert g3 == one + 2 * (one - 64 * 1024)
    assert L.fq_group_workspace_bytes(16, 0, arr(layer())) == 0
    assert L.fq_group_workspace_bytes(16, 5, arr(*[layer()] * 5)) == 0
    # larger batches run the layers in turn: the largest single workspace
    big = L.fq_group_workspace_bytes(300, 2, arr(layer(), layer(y=0x8000, C=Cg, d_out=11008)))
    assert big == max(fq.fq_workspace_bytes(300, 4096, 4512, 4512, 4096),
                      fq.fq_workspace_bytes(300, 4096, 4512, 12112, 11008))

    def fwd(a, n, ws=0x10000, nb=1 << 30, opts=None):
        return L.fq_linear_forward_group(16, n, a, ws, nb, ctypes.byref(opts) if opts else None,
                                         None)
    assert fwd(arr(layer(), layer()), 2) == 1                       # same output twice
    assert fwd(arr(layer(), layer(x=0x4000, y=0x8000)), 2) == 1     # an output is an input
    assert fwd(arr(layer(x=0x1002)), 1) == 2
    assert fwd(arr(layer()), 1, ws=0x10010) == 2
    assert fwd(arr(layer()), 1, nb=1024) == 4
    assert fwd(arr(layer()), 1, opts=fq._Opts(1, None, 0, 1000)) == 1   # no timeout hook
    assert fwd(arr(layer(ti=0x20008)), 1) == 2                       # tiles not 16-byte aligned
    assert fwd(arr(layer(to=0x20004)), 1) == 2
    # tiled operands do not change the workspace
    assert L.fq_group_workspace_bytes(16, 1, arr(layer(ti=0x20000, to=0x30000))) == \
        L.fq_group_workspace_bytes(16, 1, arr(layer()))


def test_frame_tiles_sizes_and_validation_without_gpu(L):
    # ceil(rows/128) x ceil(cols/64) tiles of 16 KiB, then 12 bytes per row tile (256-rounded)
    assert fq.fq_frame_tiles_bytes(4512, 4096) == 36 * 64 * 16384 + 512
    assert fq.fq_frame_tiles_bytes(4096, 4512) == 32 * 71 * 16384 + 512
    assert fq.fq_frame_tiles_bytes(1, 8) == 16384 + 256
    assert fq.fq_frame_tiles_bytes(12112, 11008) == 95 * 172 * 16384 + 1280
    assert fq.fq_frame_tiles_bytes(0, 64) == 0
    assert fq.fq_frame_tiles_bytes(64, 60) == 0
    nb = fq.fq_frame_tiles_bytes(64, 64)
    tile = L.fq_frame_tile
    assert tile(None, 64, 64, 0x100000, nb, None) == 1
    assert tile(0x1000, 0, 64, 0x100000, nb, None) == 1
    assert tile(0x1000, 64, 60, 0x100000, nb, None) == 2
    assert tile(0x1008, 64, 64, 0x100000, nb, None) == 2
    assert tile(0x1000, 64, 64, 0x100000, nb - 16, None) == 4
    assert tile(0x1000, 64, 64, 0x1000 + 4096, nb, None) == 1   # overlaps the source


def test_activation_rounding_modes_without_gpu(L):
    A8 = fq.FQ_BF16 | fq.FQ_ACT_BITS(8)
    # the tensor-core layout at any batch size, plus the fp32 z
    assert fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, A8) >= \
        fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, 0) + 16 * 4512 * 4
    assert fq.fq_workspace_bytes(300, 4096, 4512, 4512, 4096, A8) == \
        fq.fq_workspace_bytes(300, 4096, 4512, 4512, 4096, 0) + 300 * 4512 * 4
    assert fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, fq.FQ_ACT_BITS(1)) == 0
    assert fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096, fq.FQ_ACT_BITS(9)) == 0
    assert fq.fq_workspace_bytes(16, 4096, 4512, 4512, 4096,
                                 fq.FQ_FP32_DEBUG | fq.FQ_ACT_BITS(8)) == 0
    assert _call(L, mode=fq.FQ_ACT_BITS(9)) == 1
    assert _call(L, mode=fq.FQ_FP32_DEBUG | fq.FQ_ACT_BITS(4)) == 1
    assert _call(L, mode=1 << 20) == 1


def test_gptq_validation_without_gpu(L):
    assert fq.fq_gptq_workspace_bytes(0, 64) == 0
    n = fq.fq_gptq_workspace_bytes(12112, 4512)
    assert n >= 8 * (12112 * 4512 + 2 * 4512 * 4512) + 12112 * 4512
    assert L.fq_gptq_hessian(None, 10, 16, 0x2000, None) == 1
    assert L.fq_gptq_hessian(0x1004, 10, 16, 0x2000, None) == 2

    def q(C=0x1000, n_out=16, n_in=32, H=0x2000, damp=0.01, codes=0x3000, scale=0x4000,
          zero=0x5000, gamma=None, ws=0x10000, nb=1 << 30):
        return L.fq_quantize_gptq(C, n_out, n_in, H, damp, 0, codes, scale, zero, gamma, ws, nb,
                                  None)
    assert q(C=None) == 1
    assert q(damp=-0.5) == 1
    assert q(damp=float("nan")) == 1
    assert q(H=0x2004) == 2
    assert q(scale=0x4001) == 2
    assert q(ws=None) == 4
    assert q(ws=0x10010) == 2
    assert q(nb=1024) == 4
