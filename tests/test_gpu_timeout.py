"""The bounded-wait path of the tcgen05 kernels, made to run out on purpose
without faulting anything.

libdora_timeout_test.so is the product library rebuilt with two test hooks in
the attention kernel only: its waits give up after 5 ms instead of 1 s, and
its first CTA never issues its first K/V load (nor the bytes the stage's
barrier expects), so the S issuer's wait on that stage cannot complete and no
copy is in flight.  The kernel must raise its abort flag, let every role
leave its loop, free its tensor memory and write DORA_ERR_TIMEOUT to the
status word; the context must stay usable, so that the next call (through
the product library) is correct."""
import ctypes

import numpy as np
import pytest
import torch

import __graft_entry__ as G
import dora_synth as S
import oracle as O
import paper_2609_34325_gb300 as P
from paper_2609_34325_gb300 import build as B
from helpers import assert_close, bf, f64, i32

pytestmark = pytest.mark.gpu
DORA_ERR_TIMEOUT = 4               # include/dora.h: a bounded pipeline wait ran out


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    G.build()
    P.load_library()
    torch.cuda.set_device(0)


def _timeout_lib():
    lib = ctypes.CDLL(B.TIMEOUT_TEST_LIB_PATH)
    vp, i32_, f32_ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_float
    fn = lib.dora_varlen_attn
    fn.restype = ctypes.c_int
    fn.argtypes = [vp, vp, i32_, i32_, i32_, i32_, i32_, f32_, vp, vp, vp]
    return lib


def test_attention_wait_runs_out_reports_timeout_and_the_next_call_is_correct():
    heads = 3
    lens = np.array([197, 120, 64, 197, 5, 150, 197, 80])
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    rng = np.random.default_rng(71)
    qkv_bits = S.f32_to_bf16_bits(rng.standard_normal((t, 3 * heads * 64)))
    qkv, cu_d = bf(qkv_bits), i32(cu)
    out = torch.zeros(t, heads * 64, dtype=torch.bfloat16, device="cuda:0")
    status = torch.zeros(1, dtype=torch.int32, device="cuda:0")
    stream = torch.cuda.current_stream().cuda_stream
    lib = _timeout_lib()
    for _ in range(2):                     # twice: the kernel left nothing behind
        status.zero_()
        rc = lib.dora_varlen_attn(qkv.data_ptr(), cu_d.data_ptr(), len(lens), int(lens.max()), t,
                                  heads, 64, 0.0, out.data_ptr(), status.data_ptr(), stream)
        assert rc == 0
        torch.cuda.synchronize()           # the launch ended: every wait was bounded
        assert int(status.item()) == DORA_ERR_TIMEOUT
    # the context is intact: the product library's attention on the same
    # inputs matches the oracle
    status.zero_()
    P.dora_varlen_attn(qkv, cu_d, int(lens.max()), heads, out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert_close(f64(out), O.varlen_attention(qkv_bits, cu, heads), "attention after a timeout")
