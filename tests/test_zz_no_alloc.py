"""The allocation-free decode entry point against the regular one.

certkv_decode_attn_noalloc serves callers that cannot pass a scratch buffer
(e.g. a server plugin given only input and output tensors, or a decode loop
that must not call cudaMalloc).  Two calls in a row, through the C ABI, must
match certkv_decode_attn within the decode tolerance; a call beyond the fixed
scratch must be refused before any launch.  This file is collected last so a
failure here leaves every other test already run."""
import ctypes

import numpy as np
import pytest
import torch

import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _packed_case():
    wl = W.Workload("NA", B=1, L=2, Hq=8, H=2, n=2000, d=128, w=16, keep=(1, 8), kind="planted")
    K, V, Q = W.draw(wl, device="cuda")
    return wl, ck.certkv_compress(K, V, Q, wl.B_live)


def test_noalloc_decode_matches_regular_decode_twice():
    wl, packed = _packed_case()
    lib = ck.load_library()
    for step in (0, 1):  # two calls in a row share the static scratch
        q = W.draw_decode_queries(wl, step, device="cuda")
        ref = ck.certkv_decode_attn(q, packed, hkv=wl.H)
        out = torch.empty_like(q)
        shape = ck.certkv_shape(wl.B, wl.L, wl.Hq, wl.H, wl.n, wl.d, wl.w)
        st = packed.struct()
        rc = lib.certkv_decode_attn_noalloc(
            ctypes.byref(shape), ctypes.c_void_p(q.data_ptr()), ctypes.byref(st),
            ctypes.c_float(0.0), packed.tail_slot, ctypes.c_void_p(out.data_ptr()),
            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert rc == ck.OK, ck.certkv_strerror(rc)
        torch.cuda.synchronize()
        parity.check_decode(out, ref.float().cpu().numpy())
        np.testing.assert_array_equal(out.cpu().float().numpy(), ref.cpu().float().numpy())


def test_noalloc_decode_refuses_beyond_its_scratch():
    """The size limit is checked before the pointers: with null pointers a
    too-large call must come back ETOOLARGE, and should the size check ever let
    it through, the null pointers make it EINVAL; nothing is launched either way."""
    lib = ck.load_library()
    shape = ck.certkv_shape(8, 80, 64, 8, 32768, 128, 64)  # (B*L*H + 1024)*G = 49152
    st = ck.certkv_packed(None, None, None, None, None, 1 << 30, None, None)
    rc = lib.certkv_decode_attn_noalloc(ctypes.byref(shape), None, ctypes.byref(st),
                                        ctypes.c_float(0.0), 1, None, None)
    assert rc == ck.ETOOLARGE
    assert "fixed 16 MiB scratch" in ck.certkv_strerror(rc)
