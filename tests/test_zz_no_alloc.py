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


def test_noalloc_rejects_calls_beyond_its_scratch():
    # The buffers below are 16-byte dummies, so the call must be refused before
    # anything is launched.  The geometry is chosen so that the per-position
    # score rows alone (seven fp32 / uint32 rows per KV head and position) are far
    # beyond the 32 MiB array, whatever else the scratch holds.
    wl = synth.WORKLOADS["llama8b_l32768_b128"]
    batch, L = 16, 131072
    params = kvec.params_from_workload(wl, max_batch=batch, max_seqlen=L)
    lower_bound = batch * params.num_kv_heads * L * 4 * 7
    assert lower_bound > 8 * 32 * 2**20, "the geometry no longer exceeds the scratch by a safe margin"
    cu = torch.arange(0, (batch + 1) * L, L, dtype=torch.int32)
    dummy = torch.zeros(16, dtype=torch.uint8, device="cuda")
    p = dummy.data_ptr()
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_select_layer_noalloc(params, batch, cu.data_ptr(), cu.cuda().data_ptr(), p, p, p, p, wl.budget,
                                       p, p, p, torch.cuda.current_stream().cuda_stream)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    assert "scratch" in str(e.value)
