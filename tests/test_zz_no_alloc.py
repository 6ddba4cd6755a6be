"""kvec_select_layer_noalloc: the layer selection for callers that cannot
allocate device memory (a host that owns every allocation and forbids the
library from making its own, so kvec_create's workspace is not an option).

The entry point takes its scratch from a static device array inside libkvec.
This file is collected last so that, if it fails, a run that stops at the
first failure has already run every other test.  It passes alone in a fresh
process and after the rest of the suite.
"""
import pytest
import torch

from paper_2606_29563_gb300 import kvec, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2606_29563_gb300 import build as kbuild
    kbuild.build()


def _noalloc_layer(params, cu, x, state, budget):
    batch = cu.numel() - 1
    idx = torch.empty((batch, params.num_kv_heads, budget), dtype=torch.int32, device="cuda")
    ok = torch.empty((batch, params.num_kv_heads, budget, params.head_dim), dtype=torch.bfloat16, device="cuda")
    ov = torch.empty_like(ok)
    cu_dev = cu.cuda()
    kvec.kvec_select_layer_noalloc(params, batch, cu.data_ptr(), cu_dev.data_ptr(), x["q_obs"].data_ptr(),
                                   x["k"].data_ptr(), x["v"].data_ptr(), state.data_ptr(), budget, idx.data_ptr(),
                                   ok.data_ptr(), ov.data_ptr(), torch.cuda.current_stream().cuda_stream)
    return idx, ok, ov


def test_noalloc_matches_handle_entry_point_on_two_calls_in_a_row():
    wl = synth.small_workload(seqlens=(700, 333, 1200), layers=2, budget=96, num_ext_heads=1)
    params = kvec.params_from_workload(wl)
    layers = [{k: v.cuda() for k, v in x.items()} for x in synth.make_layers(wl, 2)]
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)

    sel = kvec.KvecSelector(params)
    st_ref = sel.new_state(wl.batch)
    ref = [[t.clone() for t in sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st_ref, wl.budget)]
           for x in layers]
    torch.cuda.synchronize()
    sel.close()

    st = torch.zeros((wl.batch, kvec.kvec_state_bytes(params.max_seqlen)), dtype=torch.uint8, device="cuda")
    got = [_noalloc_layer(params, cu, x, st, wl.budget) for x in layers]
    torch.cuda.synchronize()
    # Same kernels on the same inputs: indices, gathered rows and state agree exactly
    # (the tolerance of the parity tests is exact equality for indices, K/V and state).
    for (ri, rk, rv), (gi, gk, gv) in zip(ref, got):
        assert torch.equal(ri, gi)
        assert torch.equal(rk, gk)
        assert torch.equal(rv, gv)
    assert torch.equal(st_ref, st)
    kvec.kvec_noalloc_sync_status(torch.cuda.current_stream().cuda_stream)   # no device-side error


# (A call whose geometry exceeds the scratch array is refused before any CUDA
# call; tests/test_abi.py checks that without a GPU.)


def test_noalloc_reports_the_layer_limit_refusal():
    """n_t is 8-bit (Section 4.2's counters), so a state may count at most 255
    layers.  A call on a state that already counts 255 is refused on the device,
    leaves the state as it was, and kvec_noalloc_sync_status reports it."""
    wl = synth.small_workload(seqlens=(301,), layers=1)
    params = kvec.params_from_workload(wl)
    x = {k: v.cuda() for k, v in synth.make_layer(wl, 0).items()}
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    stream = torch.cuda.current_stream().cuda_stream
    st = torch.zeros((1, kvec.kvec_state_bytes(params.max_seqlen)), dtype=torch.uint8, device="cuda")
    st[0, 0] = 255   # layers_done, little endian
    before = st.clone()
    _noalloc_layer(params, cu, x, st, wl.budget)
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_noalloc_sync_status(stream)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    assert torch.equal(st, before)
    kvec.kvec_noalloc_sync_status(stream)   # reported once, then cleared
    st[0, 0] = 254
    _noalloc_layer(params, cu, x, st, wl.budget)
    kvec.kvec_noalloc_sync_status(stream)
    assert st[0, 0].item() == 255


def test_noalloc_reports_a_device_timeout_and_recovers():
    """A bounded device wait that gives up (forced with the test fault of the
    window kernel) is reported by kvec_noalloc_sync_status; the next call runs
    normally and matches the handle entry point."""
    wl = synth.small_workload(seqlens=(700, 333), layers=1, budget=96, num_ext_heads=1)
    params = kvec.params_from_workload(wl)
    x = {k: v.cuda() for k, v in synth.make_layer(wl, 0).items()}
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    stream = torch.cuda.current_stream().cuda_stream
    st = torch.zeros((wl.batch, kvec.kvec_state_bytes(params.max_seqlen)), dtype=torch.uint8, device="cuda")
    try:
        kvec.kvec_set_test_fault(1)
        _noalloc_layer(params, cu, x, st, wl.budget)
        with pytest.raises(kvec.KvecError) as e:
            kvec.kvec_noalloc_sync_status(stream)
        assert e.value.status == kvec.KVEC_ERR_DEVICE_TIMEOUT
    finally:
        kvec.kvec_set_test_fault(0)
    st.zero_()
    got = _noalloc_layer(params, cu, x, st, wl.budget)
    kvec.kvec_noalloc_sync_status(stream)
    sel = kvec.KvecSelector(params)
    st_ref = sel.new_state(wl.batch)
    ref = sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st_ref, wl.budget)
    torch.cuda.synchronize()
    for a, b in zip(ref, got):
        assert torch.equal(a, b)
    assert torch.equal(st_ref, st)
    sel.close()


