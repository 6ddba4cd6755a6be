"""The device-side timeout path, driven on purpose without faulting the GPU.

Every wait of the CUDA path on an mbarrier is bounded: when it gives up, the
kernel records an error word, stops issuing work, waits for the copies it has
in flight and returns, and kvec_sync_status reports KVEC_ERR_DEVICE_TIMEOUT.
kvec_set_test_fault(1) makes that happen: every window kernel withholds the
signal of its first accumulator, so its epilogue's wait (limited to about
20 us under the fault) runs out.  The test checks that the status is reported
once and cleared, and that the same handle then runs a normal layer that
matches the fp64 oracle.
"""
import pytest
import torch

import parity
from paper_2606_29563_gb300 import kvec, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2606_29563_gb300 import build as kbuild
    import oracle
    kbuild.build()
    oracle.build()


def test_window_wait_timeout_is_reported_and_the_handle_recovers():
    wl = synth.small_workload(seqlens=(700, 333), layers=2, budget=96, num_ext_heads=1)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    x = {k: v.cuda() for k, v in synth.make_layer(wl, 0).items()}
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    st = sel.new_state(wl.batch)
    kvec.kvec_sync_status(sel.handle)
    try:
        kvec.kvec_set_test_fault(1)
        sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st, wl.budget)
        with pytest.raises(kvec.KvecError) as e:
            kvec.kvec_sync_status(sel.handle)
        assert e.value.status == kvec.KVEC_ERR_DEVICE_TIMEOUT
        # A multi-layer call under the fault runs eagerly (never captured) and reports too.
        outs = [sel.alloc_outputs(wl.batch, wl.budget) for _ in range(2)]
        for _ in range(2):
            sel.select_layers(cu, cu.cuda(), [x["q_obs"]] * 2, [x["k"]] * 2, [x["v"]] * 2, st, wl.budget, outs)
            with pytest.raises(kvec.KvecError) as e:
                kvec.kvec_sync_status(sel.handle)
            assert e.value.status == kvec.KVEC_ERR_DEVICE_TIMEOUT
    finally:
        kvec.kvec_set_test_fault(0)
    kvec.kvec_sync_status(sel.handle)   # the error was cleared by the first report
    # The same handle runs normally afterwards and matches the oracle.
    errs = parity.run_parity(wl, sel=sel)
    assert not errs, "\n".join(errs[:25])
    sel.close()
