"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Every case is teacher-forced layer by layer (tests/parity.py): scores within the
2e-3 relative tolerance, kept-index sets identical outside the tie band, and
gathered K/V plus the coverage-state update bit-exact given the GPU's indices.
"""
import numpy as np
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


def _assert_parity(wl, **kw):
    errs = parity.run_parity(wl, **kw)
    assert not errs, "\n".join(errs[:25])


def test_small_two_layers():
    _assert_parity(synth.small_workload(seqlens=(700,), layers=2))


@pytest.mark.parametrize("g,Hkv", [(1, 4), (2, 4), (4, 2), (7, 4), (8, 2)])
def test_group_sizes(g, Hkv):
    _assert_parity(synth.small_workload(seqlens=(523,), num_q_heads=g * Hkv, num_kv_heads=Hkv, layers=2,
                                        num_ext_heads=1))


@pytest.mark.parametrize("L", [33, 129, 255, 256, 257, 1000])
def test_ragged_tails_and_short_sequences(L):
    # w = 32: L = 33 leaves one candidate; 129 / 257 end one token into a new tile.
    _assert_parity(synth.small_workload(seqlens=(L,), budget=48, layers=2))


def test_ragged_batch_with_keep_all_members():
    # 40 and 64 fit the budget (keep everything); the others are evicted.
    _assert_parity(synth.small_workload(seqlens=(40, 900, 64, 1531, 300), budget=64, layers=3))


def test_budget_equals_window():
    _assert_parity(synth.small_workload(seqlens=(600,), budget=32, layers=2))


@pytest.mark.parametrize("pool", [1, 3, 15])
def test_pool_widths(pool):
    _assert_parity(synth.small_workload(seqlens=(640,), pool_kernel=pool, layers=2))


@pytest.mark.parametrize("over", [dict(num_ext_heads=0, lam=0.0), dict(lam=0.0), dict(beta=0.0), dict(beta=1.0),
                                  dict(lam=2.0, beta=0.1), dict(obs_window=32, ext_window=32),
                                  dict(window=16, obs_window=8, ext_window=16)])
def test_hyperparameter_corners(over):
    _assert_parity(synth.small_workload(seqlens=(777,), layers=2, **over))


@pytest.mark.parametrize("over", [dict(pool_mode=1), dict(head_criterion=1),
                                  dict(pool_mode=1, head_criterion=1, num_ext_heads=2, pool_kernel=5),
                                  dict(window=48, obs_window=32, ext_window=48)])
def test_paper_variants(over):
    # Average pooling, the entropy head criterion (Section 5.4 ablation) and the
    # O = 32 / O' = 48 reading of the windows.
    _assert_parity(synth.small_workload(seqlens=(900, 421), layers=2, **over))


@pytest.mark.parametrize("over", [dict(pool_mode=1), dict(head_criterion=1, num_ext_heads=5)])
def test_paper_variants_with_split_head_groups(over):
    # 16 KV heads: the window kernel splits them over two CTAs per tile and the
    # heads kernel combines the groups' maxima of I before pooling.
    _assert_parity(synth.small_workload(seqlens=(700,), num_q_heads=16, num_kv_heads=16, layers=2, **over))


def test_variants_llama8b_l8192_b512_first_layers():
    wl = synth.WORKLOADS["llama8b_l8192_b512"].replace(layers=2, pool_mode=1, head_criterion=1)
    _assert_parity(wl)


def test_uniform_keys_tie_to_lowest_positions():
    """K = 0 makes every candidate score equal: selection must be the lowest positions (exact ties)."""
    wl = synth.small_workload(seqlens=(400,), budget=64, layers=1)
    params = kvec.params_from_workload(wl)
    sel = kvec.KvecSelector(params)
    x = synth.make_layer(wl, 0)
    k = torch.zeros_like(x["k"]).cuda()
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    st = sel.new_state(1)
    idx, _, _ = sel.select_layer(cu, cu.cuda(), x["q_obs"].cuda(), k, x["v"].cuda(), st, wl.budget)
    torch.cuda.synchronize()
    expect = list(range(wl.budget - wl.window)) + list(range(400 - wl.window, 400))
    for h in range(wl.num_kv_heads):
        assert idx[0, h].cpu().tolist() == expect
    sel.close()


def test_uniform_keys_long_row_tie_to_lowest_positions():
    """K = 0 on a 20000-position row: every candidate scores the same, so the
    radix select's sampled threshold finds all keys above it (far more than the
    list holds) and falls back to the full digit passes; the preserved tokens
    and the fill must still be the lowest positions."""
    L, budget = 20000, 64
    wl = synth.small_workload(seqlens=(L,), budget=budget, layers=1)
    params = kvec.params_from_workload(wl)
    sel = kvec.KvecSelector(params)
    x = synth.make_layer(wl, 0)
    k = torch.zeros_like(x["k"]).cuda()
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    st = sel.new_state(1)
    idx, _, _ = sel.select_layer(cu, cu.cuda(), x["q_obs"].cuda(), k, x["v"].cuda(), st, budget)
    torch.cuda.synchronize()
    expect = list(range(budget - wl.window)) + list(range(L - wl.window, L))
    for h in range(wl.num_kv_heads):
        assert idx[0, h].cpu().tolist() == expect
    sel.close()


@pytest.mark.parametrize("plateau,budget", [((4500, 5800), 1024), ((4800, 12000), 1024), ((5100, 5140), 64)])
def test_equal_keys_across_row_slices_tie_to_lowest_positions(plateau, budget):
    """Positions [a, b) of a 20000-position row share one key vector that every
    (constant) query favours, so their scores are equal and above every other
    candidate; B - w of them are kept, and equal keys must go to the lowest
    positions, across the warps' segments of the radix select (the row has more
    512-position segments than its 16 warps keep in registers): the kept
    candidates are one run of B - w consecutive positions starting at the
    plateau (pooling may widen it by 3).  The cases reach the threshold through
    the compacted list, the full sweep and the few-key ranking."""
    L = 20000
    wl = synth.small_workload(seqlens=(L,), budget=budget, layers=1)
    params = kvec.params_from_workload(wl)
    sel = kvec.KvecSelector(params)
    x = synth.make_layer(wl, 0)
    q = torch.full_like(x["q_obs"], 0.1).cuda()
    k = torch.zeros_like(x["k"])
    a, b = plateau
    k[a:b] = 0.5
    k = k.cuda()
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    st = sel.new_state(1)
    idx, _, _ = sel.select_layer(cu, cu.cuda(), q, k, x["v"].cuda(), st, budget)
    torch.cuda.synchronize()
    for h in range(wl.num_kv_heads):
        got = idx[0, h].cpu().tolist()
        assert got[-wl.window:] == list(range(L - wl.window, L))
        run = got[:budget - wl.window]
        assert a - 3 <= run[0] <= a + 3 and run == list(range(run[0], run[0] + len(run))), (h, run[:5], run[-5:])
    sel.close()


@pytest.mark.parametrize("kw", [dict(seqlens=(9000,), layers=3),
                                dict(seqlens=(30000,), layers=2, budget=128),
                                dict(seqlens=(17000, 600, 40), layers=3, budget=256),
                                dict(seqlens=(16384,), num_q_heads=28, num_kv_heads=4, layers=2, budget=512)])
def test_long_rows_of_small_batches_match_the_oracle(kw):
    """Few (sequence, KV head) rows of 9000 to 30000 positions over several
    layers: one to four 512-position segments per warp in the radix
    select; the ragged case adds a short sequence and one that fits the budget."""
    _assert_parity(synth.small_workload(**kw))


def test_deterministic_rerun():
    wl = synth.small_workload(seqlens=(900, 450), layers=2)
    outs = []
    for _ in range(2):
        sel = kvec.KvecSelector(kvec.params_from_workload(wl))
        cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
        st = sel.new_state(wl.batch)
        res = []
        for x in synth.make_layers(wl, 2):
            o = sel.select_layer(cu, cu.cuda(), x["q_obs"].cuda(), x["k"].cuda(), x["v"].cuda(), st, wl.budget)
            res.append([t.cpu() for t in o])
        torch.cuda.synchronize()
        res.append([st.cpu()])
        outs.append(res)
        sel.close()
    for a, b in zip(outs[0], outs[1]):
        for x, y in zip(a, b):
            assert torch.equal(x, y)


def test_graph_cache_alternating_calls_match_eager_results():
    # Two chunks of layers with different buffers, called alternately over three
    # steps: the first sighting of each runs eagerly, the second captures a
    # graph, the third replays it.  Every step must give the same indices and state.
    wl = synth.small_workload(seqlens=(900, 450), layers=4)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32).pin_memory()
    cud = cu.cuda()
    xs = [{k: v.cuda() for k, v in x.items()} for x in synth.make_layers(wl, 4)]
    outs = [sel.alloc_outputs(wl.batch, wl.budget) for _ in range(4)]
    st = sel.new_state(wl.batch)
    stream = torch.cuda.current_stream()
    steps = []
    for _ in range(3):
        kvec.kvec_reset(sel.handle, st.data_ptr(), wl.batch, stream.cuda_stream)
        for ls in ([0, 1], [2, 3]):
            sel.select_layers(cu, cud, [xs[l]["q_obs"] for l in ls], [xs[l]["k"] for l in ls],
                              [xs[l]["v"] for l in ls], st, wl.budget, [outs[l] for l in ls], stream)
        kvec.kvec_sync_status(sel.handle)
        steps.append([o[0].cpu() for o in outs] + [o[1].cpu() for o in outs] + [st.cpu()])
    for later in steps[1:]:
        for x, y in zip(steps[0], later):
            assert torch.equal(x, y)


def test_multi_layer_call_matches_layer_by_layer():
    wl = synth.small_workload(seqlens=(1100, 700), layers=4, budget=96)
    layers = [{k: v.cuda() for k, v in x.items()} for x in synth.make_layers(wl, 4)]
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    st1 = sel.new_state(wl.batch)
    one = [sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st1, wl.budget) for x in layers]
    st2 = sel.new_state(wl.batch)
    many = [sel.alloc_outputs(wl.batch, wl.budget) for _ in layers]
    sel.select_layers(cu, cu.cuda(), [x["q_obs"] for x in layers], [x["k"] for x in layers],
                      [x["v"] for x in layers], st2, wl.budget, many)
    torch.cuda.synchronize()
    for a, b in zip(one, many):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
    assert torch.equal(st1, st2)
    sel.close()


# ---- window-row log-sum-exp supplied by the caller (no statistics pass) ----

@pytest.mark.parametrize("kw", [dict(seqlens=(700,), layers=2),
                                dict(seqlens=(40, 900, 64, 1531), budget=64, layers=2),
                                dict(seqlens=(523,), num_q_heads=28, num_kv_heads=4, layers=2)])
def test_lse_input_matches_the_oracle(kw):
    _assert_parity(synth.small_workload(**kw), with_lse=True)


def test_lse_input_llama8b_l8192_b512_first_layers():
    _assert_parity(synth.WORKLOADS["llama8b_l8192_b512"], layers=2, with_lse=True)


def test_lse_input_llama8b_ragged8_b256_first_layers():
    # The ragged batch of 8 runs the tile-owning window kernel, which takes units
    # of three candidate tiles when the caller supplies the log-sum-exp.
    _assert_parity(synth.WORKLOADS["llama8b_ragged8_b256"], layers=2, with_lse=True)


def test_lse_multi_layer_call_matches_layer_by_layer():
    wl = synth.small_workload(seqlens=(1100, 700), layers=3, budget=96)
    cpu_layers = synth.make_layers(wl, 3)
    layers = [{k: v.cuda() for k, v in x.items()} for x in cpu_layers]
    lses = [torch.from_numpy(parity.window_lse(wl, x).astype(np.float32)).cuda() for x in cpu_layers]
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    st1 = sel.new_state(wl.batch)
    one = [sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st1, wl.budget, lse=e)
           for x, e in zip(layers, lses)]
    st2 = sel.new_state(wl.batch)
    many = [sel.alloc_outputs(wl.batch, wl.budget) for _ in layers]
    sel.select_layers(cu, cu.cuda(), [x["q_obs"] for x in layers], [x["k"] for x in layers],
                      [x["v"] for x in layers], st2, wl.budget, many, lses=lses)
    torch.cuda.synchronize()
    for a, b in zip(one, many):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
    assert torch.equal(st1, st2)
    with pytest.raises(kvec.KvecError) as e:   # a misaligned lse pointer is refused before any launch
        kvec.kvec_select_layer_lse(sel.handle, wl.batch, cu.data_ptr(), cu.cuda().data_ptr(),
                                   layers[0]["q_obs"].data_ptr(), layers[0]["k"].data_ptr(),
                                   layers[0]["v"].data_ptr(), lses[0].data_ptr() + 2, st2.data_ptr(), wl.budget,
                                   *[t.data_ptr() for t in many[0]], torch.cuda.current_stream().cuda_stream)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    sel.close()


def test_layer_limit_refuses_the_whole_call_and_positions_past_L_stay_zero():
    """n_t is 8-bit, so no state may count more than 255 layers (Section 4.2's
    counters).  A call that would pass the limit reports it and leaves the state
    as it was, whichever of its layers would have crossed it; a call that ends at
    255 runs.  Positions from L on (here L = 301, not a multiple of 4, in a state
    sized for 400) are never written."""
    L, ML = 301, 400
    wl = synth.small_workload(seqlens=(L,), layers=2)
    layers = [{k: v.cuda() for k, v in x.items()} for x in synth.make_layers(wl, 2)]
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl, max_seqlen=ML))
    st = sel.new_state(1)
    st[0, 0] = 254   # layers_done, little endian
    before = st.clone()
    outs = [sel.alloc_outputs(1, wl.budget) for _ in layers]
    sel.select_layers(cu, cu.cuda(), [x["q_obs"] for x in layers], [x["k"] for x in layers],
                      [x["v"] for x in layers], st, wl.budget, outs)
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_sync_status(sel.handle)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    assert torch.equal(st, before)
    x = layers[0]
    sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st, wl.budget)
    kvec.kvec_sync_status(sel.handle)
    s = st.cpu()
    assert s[0, 0].item() == 255 and s[0, 4:8].view(torch.int32).item() == L
    n = s[0, 16:16 + ((ML + 15) // 16) * 16]
    assert int(n[:L].sum()) > 0 and not n[L:].any()
    sel.close()


def test_call_validation_on_device():
    wl = synth.small_workload(seqlens=(300,))
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    x = {k: v.cuda() for k, v in synth.make_layer(wl, 0).items()}
    st = sel.new_state(1)
    cu_ok = torch.tensor([0, 300], dtype=torch.int32)
    cases = [
        (torch.tensor([0, 20], dtype=torch.int32), wl.budget),     # L < w
        (torch.tensor([0, 301], dtype=torch.int32), wl.budget),    # L > max_seqlen
        (torch.tensor([1, 300], dtype=torch.int32), wl.budget),    # cu[0] != 0
        (cu_ok, wl.window - 1),                                    # B < w
    ]
    for cu, budget in cases:
        with pytest.raises(kvec.KvecError) as e:
            sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st, budget)
        assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    with pytest.raises(kvec.KvecError):   # misaligned K, refused by the host checks
        kvec.kvec_select_layer(
            sel.handle, 1, cu_ok.data_ptr(), cu_ok.cuda().data_ptr(), x["q_obs"].data_ptr(), x["k"].data_ptr() + 2,
            x["v"].data_ptr(), st.data_ptr(), wl.budget, *[t.data_ptr() for t in sel.alloc_outputs(1, wl.budget)],
            torch.cuda.current_stream().cuda_stream)
    assert st.cpu().sum().item() == 0   # rejected calls launched nothing
    sel.close()


# ---- the five workloads at full size (teacher-forced, a few layers each) ----

def test_mha8_l1024_b128_full():
    _assert_parity(synth.WORKLOADS["mha8_l1024_b128"])


def test_llama8b_l8192_b512_all_layers():
    # All 32 layers, so the late layers (n_t up to 31, coverage near 1, focus
    # near 0) are compared too.
    _assert_parity(synth.WORKLOADS["llama8b_l8192_b512"], layers=32)


def test_llama8b_l32768_b128_first_layers():
    _assert_parity(synth.WORKLOADS["llama8b_l32768_b128"], layers=2)


def test_llama8b_ragged8_b256_first_layers():
    _assert_parity(synth.WORKLOADS["llama8b_ragged8_b256"], layers=2)


@pytest.mark.parametrize("budget", synth.QWEN_BUDGETS)
def test_qwen7b_l16384_budget_sweep(budget):
    _assert_parity(synth.WORKLOADS["qwen7b_l16384_b512"].replace(budget=budget), layers=2)


# ---- top-B over every position (all_positions = 1, Section 4.1 read literally) ----

@pytest.mark.parametrize("kw", [dict(seqlens=(900, 421), layers=2),
                                dict(seqlens=(40, 1000, 64, 257), budget=64, layers=2),
                                dict(seqlens=(777,), budget=20, layers=2),
                                dict(seqlens=(523,), num_q_heads=28, num_kv_heads=4, layers=2),
                                dict(seqlens=(700,), num_q_heads=16, num_kv_heads=16, layers=2),
                                dict(seqlens=(640,), pool_mode=1, head_criterion=1, layers=2),
                                dict(seqlens=(600,), window=48, obs_window=32, ext_window=48, layers=2)])
def test_all_positions_matches_the_oracle(kw):
    # Candidates [0, L): the window part scored with its causal attention (a
    # token there is seen only by the later window rows), nothing kept by rule;
    # a budget below the window, keep-all members, split head groups, the variants.
    _assert_parity(synth.small_workload(all_positions=1, **kw))


def test_all_positions_with_caller_lse():
    _assert_parity(synth.small_workload(seqlens=(1100, 333), layers=2, all_positions=1), with_lse=True)


def test_all_positions_llama8b_l8192_b512_first_layers():
    _assert_parity(synth.WORKLOADS["llama8b_l8192_b512"].replace(all_positions=1), layers=2)


def test_all_positions_multi_layer_call_matches_layer_by_layer():
    wl = synth.small_workload(seqlens=(1100, 700), layers=3, budget=96, all_positions=1)
    layers = [{k: v.cuda() for k, v in x.items()} for x in synth.make_layers(wl, 3)]
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    st1 = sel.new_state(wl.batch)
    one = [sel.select_layer(cu, cu.cuda(), x["q_obs"], x["k"], x["v"], st1, wl.budget) for x in layers]
    st2 = sel.new_state(wl.batch)
    many = [sel.alloc_outputs(wl.batch, wl.budget) for _ in layers]
    stream = torch.cuda.current_stream().cuda_stream
    for _ in range(3):   # the second call captures the pipeline, the third replays the graph
        kvec.kvec_reset(sel.handle, st2.data_ptr(), wl.batch, stream)
        sel.select_layers(cu, cu.cuda(), [x["q_obs"] for x in layers], [x["k"] for x in layers],
                          [x["v"] for x in layers], st2, wl.budget, many)
    torch.cuda.synchronize()
    for a, b in zip(one, many):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
    assert torch.equal(st1, st2)
    sel.close()


# ---- head-wise adaptive fill (a floor per head, the rest ranked over the heads) ----

@pytest.mark.parametrize("kw", [dict(seqlens=(900,), ada_floor=0.25),
                                dict(seqlens=(40, 1100, 64, 700), budget=96, ada_floor=0.2),
                                dict(seqlens=(523,), num_q_heads=28, num_kv_heads=4, ada_floor=0.0),
                                dict(seqlens=(640,), num_q_heads=16, num_kv_heads=8, ada_floor=0.5, budget=48),
                                dict(seqlens=(700, 333), ada_floor=0.2, all_positions=1)])
def test_adaptive_fill_matches_the_oracle(kw):
    kw.setdefault("num_q_heads", 16)
    kw.setdefault("num_kv_heads", 4)
    _assert_parity(synth.small_workload(head_budget=1, layers=3, **kw))


def test_adaptive_fill_with_floor_one_is_the_uniform_fill():
    """ada_floor = 1: every head ranks its whole fill itself, so indices, K/V and
    state equal the uniform fill's bit for bit."""
    wl = synth.small_workload(seqlens=(1100, 300, 700), num_q_heads=16, num_kv_heads=4, layers=2, budget=96)
    outs = []
    for hb in (0, 1):
        w = wl.replace(head_budget=hb, ada_floor=1.0)
        sel = kvec.KvecSelector(kvec.params_from_workload(w))
        cu = torch.tensor(w.cu_seqlens, dtype=torch.int32)
        st = sel.new_state(w.batch)
        res = [[t.cpu() for t in sel.select_layer(cu, cu.cuda(), x["q_obs"].cuda(), x["k"].cuda(), x["v"].cuda(),
                                                  st, w.budget)] for x in synth.make_layers(w, 2)]
        torch.cuda.synchronize()
        outs.append((res, st.cpu()))
        sel.close()
    for a, b in zip(outs[0][0], outs[1][0]):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
    assert torch.equal(outs[0][1], outs[1][1])


def test_adaptive_fill_llama8b_l8192_b512_first_layers():
    _assert_parity(synth.WORKLOADS["llama8b_l8192_b512"].replace(head_budget=1, ada_floor=0.2), layers=3)


def test_adaptive_fill_llama8b_ragged8_b256_first_layers():
    _assert_parity(synth.WORKLOADS["llama8b_ragged8_b256"].replace(head_budget=1, ada_floor=0.2), layers=2)


def _random_small_workload(i):
    """A seeded random configuration inside the kernels' limits (d = 128, g*w a
    multiple of 8 and <= 256, odd pool width <= 15): batch, lengths, heads,
    windows, pooling, delta, lambda, beta, budget and the variants at random."""
    rng = np.random.default_rng(5000 + i)
    Hkv = int(rng.choice([1, 2, 4, 8]))
    g = int(rng.choice([1, 2, 3, 4, 7, 8]))
    w = int(rng.choice([8, 16, 24, 32]))
    O = int(rng.integers(1, w + 1))
    Oe = int(rng.integers(O, w + 1))
    batch = int(rng.integers(1, 4))
    seqlens = tuple(int(x) for x in rng.integers(w, 1201, size=batch))
    all_positions = int(rng.random() < 0.25)
    head_budget = int(rng.random() < 0.25)
    return synth.small_workload(
        name=f"random{i}", seqlens=seqlens, num_q_heads=g * Hkv, num_kv_heads=Hkv, window=w, obs_window=O,
        ext_window=Oe, pool_kernel=int(rng.choice([1, 3, 7, 15])), num_ext_heads=int(rng.integers(0, Hkv + 1)),
        lam=float(rng.choice([0.0, 1.0, 2.0])), beta=float(rng.choice([0.0, 0.25, 0.5])),
        budget=int(rng.integers(1 if all_positions else w, 301)), layers=2, seed=5000 + i,
        pool_mode=int(rng.random() < 0.25), head_criterion=int(rng.random() < 0.25), all_positions=all_positions,
        head_budget=head_budget, ada_floor=float(rng.choice([0.0, 0.2, 0.5])) if head_budget else 1.0)


@pytest.mark.parametrize("i", range(16))
def test_random_small_configurations_match_the_oracle(i):
    _assert_parity(_random_small_workload(i))
