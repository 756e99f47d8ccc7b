"""The tensor-core kernel's bounded waits, made to run out on purpose.

Every mbarrier wait of the tensor-core decode gives up after a bounded number
of polls: the thread raises the CTA's abort flag and the status word, every
warp of the CTA skips its remaining work, the issuing warps wait (bounded)
for the MMAs and TMA copies they started, and tensor memory is freed.  The
test hook pic_decode_test_wait_fault makes one decoding thread of the first
CTA withhold one arrival and cuts the poll limit to microseconds' worth, so
that the issuing warp's wait runs out; nothing faults, traps or hangs.

Checked: the call reports PIC_ERR_TIMEOUT (through the handle, and through
the allocation-free entry point's status read), the flag is then clear, and
the next normal decode on the same handle, or through the same static status
word, matches the oracle (the aborted launch freed its tensor memory and left
nothing behind).  Both kernel organisations run: the output layer on the
tensor cores with per-thread latent copies (7-64-64-3), and on the CUDA cores
with TMA-staged rows (16-64-64-64-3 GELU).
"""
import numpy as np
import pytest

from paper_2609_09020_gb300 import workloads as wk

from decode_util import max_abs_diff, oracle_full

pytestmark = pytest.mark.gpu
P = "fp16_tc"
SHORT_LIMIT = 1 << 10  # polls before a wait gives up while the fault is on


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_09020_gb300 import build
    build.build()


CASES = [
    (wk.custom("abort_a", 64, 256, 7, 1, (7, 64, 64, 3), weight_dtype="fp16", precisions=(P,)),
     "copies"),
    (wk.custom("abort_b", 48, 384, 8, 2, (16, 64, 64, 64, 3), act="gelu", clip=63, lap_scale=4.0,
               precisions=(P,)), "tma"),
]


def _buffers(wl, x):
    import torch
    dev = torch.device("cuda:0")
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    out = torch.full((x.latents.shape[0], 3, wl.H, wl.W), float("nan"), device=dev)
    return t(x.latents), t(x.steps), t(x.weights_for(P)), out


@pytest.mark.parametrize("wl,staging", CASES, ids=lambda c: getattr(c, "name", c))
def test_withheld_arrival_times_out_and_the_handle_recovers(orc, wl, staging):
    import torch
    from paper_2609_09020_gb300 import pic
    x = wk.make_inputs(wl)
    lat, st, w, out = _buffers(wl, x)
    dec = pic.Decoder.for_workload(wl, P, staging=staging)
    assert ("_tma" in dec.kernel_name) == (staging == "tma")
    s = torch.cuda.current_stream().cuda_stream
    try:
        assert pic.pic_decode_test_wait_fault(1, SHORT_LIMIT) == pic.PIC_OK
        rc = pic.pic_decode_batch(dec.handle, 1, lat.data_ptr(), st.data_ptr(), w.data_ptr(), wl.H,
                                  wl.W, out.data_ptr(), s)
        assert rc == pic.PIC_OK
        assert pic.pic_decode_check(dec.handle, s) == pic.PIC_ERR_TIMEOUT
    finally:
        pic.pic_decode_test_wait_fault(0, 0)
    assert pic.pic_decode_check(dec.handle, s) == pic.PIC_OK  # the flag was cleared
    # the same handle decodes normally afterwards
    dec.decode_batch(lat, st, w, wl.H, wl.W, out, B=1)
    dec.check()
    got = out.cpu().numpy()[0]
    d, where = max_abs_diff(got, oracle_full(orc, wl, x, 0, P))
    assert d <= 2e-4, (d, where)
    dec.close()


def test_noalloc_status_read_reports_the_timeout(orc):
    import torch
    from paper_2609_09020_gb300 import pic
    wl, _ = CASES[0]
    x = wk.make_inputs(wl)
    lat, st, w, out = _buffers(wl, x)
    arch = pic.make_arch(wl.L, wl.C, wl.dims, wl.act, P, True, wl.H, wl.W, 1)
    s = torch.cuda.current_stream().cuda_stream
    assert pic.pic_decode_noalloc_check(s) == pic.PIC_OK
    try:
        pic.pic_decode_test_wait_fault(1, SHORT_LIMIT)
        rc = pic.pic_decode_batch_noalloc(arch, 1, lat.data_ptr(), st.data_ptr(), w.data_ptr(),
                                          wl.H, wl.W, out.data_ptr(), s)
        assert rc == pic.PIC_OK
        assert pic.pic_decode_noalloc_check(s) == pic.PIC_ERR_TIMEOUT
    finally:
        pic.pic_decode_test_wait_fault(0, 0)
    assert pic.pic_decode_noalloc_check(s) == pic.PIC_OK
    rc = pic.pic_decode_batch_noalloc(arch, 1, lat.data_ptr(), st.data_ptr(), w.data_ptr(), wl.H,
                                      wl.W, out.data_ptr(), s)
    assert rc == pic.PIC_OK and pic.pic_decode_noalloc_check(s) == pic.PIC_OK
    d, where = max_abs_diff(out.cpu().numpy()[0], oracle_full(orc, wl, x, 0, P))
    assert d <= 2e-4, (d, where)


def test_hook_rejects_bad_arguments():
    from paper_2609_09020_gb300 import pic
    assert pic.pic_decode_test_wait_fault(2, 0) == pic.PIC_ERR_INVALID_ARG
    assert pic.pic_decode_test_wait_fault(0, 0) == pic.PIC_OK
