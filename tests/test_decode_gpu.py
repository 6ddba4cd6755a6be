"""GPU parity of one decoding step over the compacted cache (kvec_decode_attention,
through the C ABI) against the fp64 oracle (oracle/decode.py).

Tolerance, per output row: |gpu - oracle| <= 2e-5 * max_j |v_j| + 1e-7, v_j the
head's cached value rows.  The logits are fp32 sums of exact bf16 products
(errors of order 1e-6 in the exponent), the weights come from ex2.approx
(relative error about 2^-22) and the fp32 accumulation over the rows adds about
1e-6 relatively; the output is a convex combination of the v_j, so its error
stays near 1e-6 * max|v|.  Dropping, duplicating or misweighting one of n <= 8192
cached rows moves the output by about max|v| / n >= 1.2e-4 * max|v|, well above
the bound.
"""
import numpy as np
import pytest
import torch

from oracle.decode import decode_attention as oracle_decode
from paper_2606_29563_gb300 import kvec, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2606_29563_gb300 import build as kbuild
    kbuild.build()


def _selector(Hq, Hkv, max_batch=4, window=32):
    ow = min(16, window)
    return kvec.KvecSelector(kvec.make_params(Hq, Hkv, window=window, obs_window=ow, ext_window=window,
                                              num_ext_heads=min(3, Hkv), max_batch=max_batch, max_seqlen=1024,
                                              max_layers=4))


def _check(sel, q, k, v, lens, scale=None):
    """q [b][Hq][d], k/v [b][Hkv][cap][d] bf16 on the device; lens list."""
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    out = sel.decode_attention(q, k, v, lens_d)
    torch.cuda.synchronize()
    d = q.shape[-1]
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    f64 = lambda x: x.float().cpu().numpy().astype(np.float64)
    ref = oracle_decode(f64(q), f64(k), f64(v), lens, scale)
    got = out.cpu().numpy().astype(np.float64)
    g = q.shape[1] // k.shape[1]
    vv = f64(v)
    errs = []
    for b in range(q.shape[0]):
        n = min(max(lens[b], 0), k.shape[2])
        for hq in range(q.shape[1]):
            vmax = np.abs(vv[b, hq // g, :n]).max() if n else 0.0
            tol = 2e-5 * vmax + 1e-7
            diff = np.abs(got[b, hq] - ref[b, hq]).max()
            if not diff <= tol:
                errs.append(f"b={b} hq={hq} n={n}: max diff {diff:.3e} > tol {tol:.3e}")
    assert not errs, "\n".join(errs[:20])
    return out


def _rand(shape, gen, std=1.0):
    return (torch.randn(shape, generator=gen) * std).to(torch.bfloat16).cuda()


@pytest.mark.parametrize("batch,Hq,Hkv,cap,lens", [
    (1, 4, 4, 1, [1]),
    (2, 8, 4, 5, [5, 3]),
    (1, 32, 8, 63, [63]),
    (1, 32, 8, 64, [64]),
    (2, 32, 8, 65, [65, 1]),
    (3, 28, 4, 200, [200, 0, 137]),      # g = 7; an empty cache row gives zeros
    (2, 16, 2, 512, [512, 300]),         # g = 8
    (1, 8, 8, 1000, [999]),              # g = 1
])
def test_matches_the_oracle(batch, Hq, Hkv, cap, lens):
    gen = torch.Generator().manual_seed(cap * 131 + Hq)
    sel = _selector(Hq, Hkv)
    q = _rand((batch, Hq, 128), gen)
    k = _rand((batch, Hkv, cap, 128), gen)
    v = _rand((batch, Hkv, cap, 128), gen)
    out = _check(sel, q, k, v, lens)
    if 0 in lens:
        assert torch.all(out[lens.index(0)] == 0)


@pytest.mark.parametrize("cap,n", [(4096, 4096), (8192, 8191), (20000, 19001)])
def test_long_caches_span_several_tiles_per_split(cap, n):
    # cap > 64 * 64: each split streams several 64-row tiles (online rescaling).
    gen = torch.Generator().manual_seed(cap)
    sel = _selector(32, 8, max_batch=1)
    q = _rand((1, 32, 128), gen, std=2.0)
    k = _rand((1, 8, cap, 128), gen)
    v = _rand((1, 8, cap, 128), gen)
    _check(sel, q, k, v, [n])


def test_peaked_softmax_and_garbage_past_lens():
    gen = torch.Generator().manual_seed(7)
    sel = _selector(8, 2)
    q = _rand((2, 8, 128), gen, std=6.0)              # logits of tens: one row dominates
    k = _rand((2, 2, 300, 128), gen)
    v = _rand((2, 2, 300, 128), gen)
    lens = [177, 300]
    k[0, :, 177:] = 100.0                              # never read
    v[0, :, 177:] = float("nan")
    out = _check(sel, q, k, v, lens)
    assert torch.isfinite(out).all()


def _decode_after_selection(name, layer=0):
    """Select a layer of the named workload on the GPU, then decode one step over
    its compacted cache with lens = min(L_s, B) and compare with the oracle."""
    wl = synth.WORKLOADS[name]
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    x = synth.make_layer(wl, layer, "cuda")
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    st = sel.new_state(wl.batch)
    _, ok, ov = sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st, wl.budget)
    # The step's query: the last window row of every sequence (post-RoPE in a model).
    q = x["q_obs"][:, -1].contiguous()
    lens = [min(int(cu[b + 1] - cu[b]), wl.budget) for b in range(wl.batch)]
    _check(sel, q, ok, ov, lens)


def test_after_selection_llama8b_l8192_b512():
    _decode_after_selection("llama8b_l8192_b512")


def test_after_selection_llama8b_ragged8_b256():
    _decode_after_selection("llama8b_ragged8_b256")


def test_after_selection_qwen7b_group_of_seven():
    _decode_after_selection("qwen7b_l16384_b512")


def test_call_validation():
    sel = _selector(8, 2, max_batch=2)
    q = torch.zeros((2, 8, 128), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((2, 2, 16, 128), dtype=torch.bfloat16, device="cuda")
    lens = torch.full((2,), 16, dtype=torch.int32, device="cuda")
    out = torch.empty((2, 8, 128), dtype=torch.float32, device="cuda")
    h = sel.handle
    bad = [
        dict(batch=3), dict(batch=0), dict(cap=0), dict(cap=(1 << 20) + 1),
        dict(q=q.data_ptr() + 2), dict(k=k.data_ptr() + 8), dict(lens=lens.data_ptr() + 2), dict(q=0),
    ]
    base = dict(batch=2, q=q.data_ptr(), k=k.data_ptr(), v=k.data_ptr(), lens=lens.data_ptr(), cap=16,
                out=out.data_ptr())
    for b in bad:
        a = {**base, **b}
        with pytest.raises(kvec.KvecError) as e:
            kvec.kvec_decode_attention(h, a["batch"], a["q"], a["k"], a["v"], a["lens"], a["cap"], a["out"], 0)
        assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    wide = kvec.KvecSelector(kvec.make_params(32, 2, window=16, obs_window=8, ext_window=16, num_ext_heads=1,
                                              max_batch=1, max_seqlen=256))
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_decode_attention(wide.handle, 1, q.data_ptr(), k.data_ptr(), k.data_ptr(), lens.data_ptr(), 16,
                                   out.data_ptr(), 0)
    assert e.value.status == kvec.KVEC_ERR_UNSUPPORTED
