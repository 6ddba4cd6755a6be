"""The configuration the benchmark times: one kvec_select_layers call over every
layer of a prefill.

Inside such a call the library pipelines the layers over several streams: the
per-layer score arrays cycle through a ring of eight slots (a 32-layer call
wraps it four times, so the waits before a slot is reused run), the two
score-statistics buffers alternate, and a call repeated with the same
arguments is captured once and then replayed as a CUDA graph.  Algorithm 1
carries the coverage counts n_t from layer to layer, so a race anywhere in
that ring would change every later layer.  Each test runs the full call three
times (eager, captured, replayed) and requires every layer's kept indices,
gathered K/V rows and the final coverage state to be bit-identical to 32
single-layer calls on the same inputs.  (The single-layer calls are compared
with the fp64 oracle in test_parity_gpu.py, over all 32 layers of the same
workload.)
"""
import math

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


def _window_lse(wl, x):
    """fp32 log-sum-exp of every window query row over the keys it sees, [batch][w][H_q]:
    an input of kvec_select_layers_lse (its accuracy does not matter here, both
    sides of the comparison take the same values)."""
    w, Hq, Hkv, d = wl.window, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    g = Hq // Hkv
    out = torch.empty(wl.batch, w, Hq, dtype=torch.float32, device="cuda")
    cu = wl.cu_seqlens
    for s in range(wl.batch):
        L = cu[s + 1] - cu[s]
        q = x["q_obs"][s].float()
        k = x["k"][cu[s]:cu[s + 1]].float().repeat_interleave(g, dim=1)
        logits = torch.einsum("qhd,thd->hqt", q, k) / math.sqrt(d)
        hidden = torch.arange(L, device="cuda")[None, :] > (L - w + torch.arange(w, device="cuda"))[:, None]
        logits.masked_fill_(hidden[None], float("-inf"))
        out[s] = torch.logsumexp(logits, dim=2).transpose(0, 1)
    return out


def _check_full_call(wl, with_lse=False):
    n = wl.layers
    structure = [synth.salient_structure(wl, b, n) for b in range(wl.batch)]
    xs = [synth.make_layer(wl, l, "cuda", structure) for l in range(n)]
    lses = [_window_lse(wl, x) for x in xs] if with_lse else None
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32).pin_memory()
    cud = cu.cuda()
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    stream = torch.cuda.current_stream()

    # Reference: one call per layer, each through the one-layer pipeline.
    st_ref = sel.new_state(wl.batch)
    ref = []
    for l, x in enumerate(xs):
        o = sel.select_layer(cu, cud, x["q_obs"], x["k"], x["v"], st_ref, wl.budget,
                             lse=lses[l] if with_lse else None)
        ref.append(tuple(t.clone() for t in o))
    kvec.kvec_sync_status(sel.handle)

    outs = [sel.alloc_outputs(wl.batch, wl.budget) for _ in range(n)]
    st = sel.new_state(wl.batch)
    for rep in ("eager", "captured", "replayed"):
        for o in outs:
            for t in o:
                t.fill_(-7 if t.dtype == torch.int32 else 7)   # stale values must not survive
        kvec.kvec_reset(sel.handle, st.data_ptr(), wl.batch, stream.cuda_stream)
        sel.select_layers(cu, cud, [x["q_obs"] for x in xs], [x["k"] for x in xs], [x["v"] for x in xs], st,
                          wl.budget, outs, stream, lses=lses)
        kvec.kvec_sync_status(sel.handle)
        for l in range(n):
            for name, a, b in zip(("out_idx", "out_k", "out_v"), ref[l], outs[l]):
                assert torch.equal(a, b), f"{rep} call: layer {l} {name} differs from the layer-by-layer calls"
        assert torch.equal(st_ref, st), f"{rep} call: coverage state differs from the layer-by-layer calls"
    hdr = st.cpu()[:, :4].contiguous().view(torch.int32)
    assert (hdr[:, 0] == n).all()
    sel.close()


def test_full_call_llama8b_l8192_b512():
    _check_full_call(synth.WORKLOADS["llama8b_l8192_b512"])


def test_full_call_llama8b_ragged8_b256():
    _check_full_call(synth.WORKLOADS["llama8b_ragged8_b256"])


def test_full_call_llama8b_l8192_b512_with_caller_lse():
    _check_full_call(synth.WORKLOADS["llama8b_l8192_b512"], with_lse=True)


def test_full_call_llama8b_ragged8_b256_with_caller_lse():
    _check_full_call(synth.WORKLOADS["llama8b_ragged8_b256"], with_lse=True)


def test_full_call_llama8b_l8192_b512_all_positions():
    _check_full_call(synth.WORKLOADS["llama8b_l8192_b512"].replace(all_positions=1))


def test_full_call_qwen7b_l16384_b2048():
    # 28 layers, 4 KV heads (group 7), the largest budget of the sweep.
    _check_full_call(synth.WORKLOADS["qwen7b_l16384_b512"].replace(budget=2048))


def test_full_call_llama8b_l8192_b512_adaptive_fill():
    # The joint ranking of every head's fill runs after each layer's selection
    # on the chain stream, in the captured graph as a programmatic dependent.
    _check_full_call(synth.WORKLOADS["llama8b_l8192_b512"].replace(head_budget=1, ada_floor=0.2))
