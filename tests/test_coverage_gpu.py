"""Coverage read from the GPU's coverage state (paper_2606_29563_gb300.coverage)
against the fp64 oracle's count of covered tokens, one layer per method and
budget so that both sides start from the same state."""
import pytest
import torch

import oracle
from paper_2606_29563_gb300 import coverage, kvec, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2606_29563_gb300 import build as kbuild
    kbuild.build()
    oracle.build()


@pytest.mark.parametrize("method", sorted(coverage.METHODS))
@pytest.mark.parametrize("rate", [0.5, 0.9])
def test_one_layer_coverage_matches_the_oracle(method, rate):
    base = synth.small_workload(seqlens=(700, 421), layers=1)
    L_min = min(base.seqlens)
    wl = base.replace(budget=max(base.window, int(round((1 - rate) * L_min))), **coverage.METHODS[method])
    x = synth.make_layer(wl, 0)
    sel = kvec.KvecSelector(kvec.params_from_workload(wl))
    cu = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    st = sel.new_state(wl.batch)
    sel.select_layer(cu, cu.cuda(), x["q_obs"].cuda(), x["k"].cuda(), x["v"].cuda(), st, wl.budget)
    kvec.kvec_sync_status(sel.handle)
    got = coverage.coverage_of_state(st.cpu(), wl.seqlens)
    r = oracle.select_layer(oracle.OracleParams.from_workload(wl), wl.cu_seqlens, x["q_obs"], x["k"], x["v"],
                            oracle.new_state(wl.batch, wl.max_seqlen), wl.budget, max_seqlen=wl.max_seqlen)
    expect = [int(r["coverage"][b]) / L for b, L in enumerate(wl.seqlens)]
    for b, L in enumerate(wl.seqlens):
        # Identical selections give identical counts; a token swapped inside the
        # score tie band may move the count by one per head.
        assert abs(got[b] - expect[b]) * L <= wl.num_kv_heads, (b, got[b], expect[b])


def test_sweep_reports_every_rate_and_method():
    wl = synth.small_workload(seqlens=(600,), layers=3)
    res = coverage.sweep(wl, rates=(0.25, 0.75))
    assert res["budgets"] == [max(wl.window, round(0.75 * 600)), max(wl.window, round(0.25 * 600))]
    assert res["checkpoints"] == [1, 2, 3]
    for m in coverage.METHODS:
        assert len(res["coverage"][m]) == 2
        for per_layer in res["coverage"][m]:
            assert len(per_layer) == 3 and all(0.0 < c <= 1.0 for c in per_layer)
            # n_t only grows: coverage never falls as layers are added.
            assert per_layer == sorted(per_layer)
        assert res["drop"][m] == [c[-1] - 1.0 for c in res["coverage"][m]]
