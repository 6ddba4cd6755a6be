"""Host-side checks of the C ABI that need no GPU: the library builds and loads,
exports every entry point include/kvec.h declares, sizes the coverage state like
the oracle, and rejects bad arguments before touching CUDA."""
import ctypes
import os
import re

import pytest

import oracle
from paper_2606_29563_gb300 import build as kbuild
from paper_2606_29563_gb300 import kvec

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    kbuild.build()
    return kvec.load()


def declared_entry_points():
    text = open(os.path.join(ROOT, "include", "kvec.h")).read()
    return sorted(set(re.findall(r"KVEC_API\s+[\w\s\*]+?\b(kvec_\w+)\s*\(", text)))


def test_header_declares_expected_entry_points():
    names = declared_entry_points()
    assert set(names) == set(kvec.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    raw = ctypes.CDLL(kvec.LIB_PATH)
    for name in declared_entry_points():
        assert hasattr(raw, name), name


def test_state_bytes_matches_oracle(lib):
    for ml in (1, 31, 32, 33, 1000, 8192, 16384, 32768, 131072):
        assert kvec.kvec_state_bytes(ml) == oracle.state_bytes(ml)
        assert kvec.kvec_state_bytes(ml) % 16 == 0
    assert kvec.kvec_state_bytes(0) == 0


BAD_PARAMS = [
    (dict(num_q_heads=30, num_kv_heads=8), kvec.KVEC_ERR_INVALID_ARG),
    (dict(num_kv_heads=0), kvec.KVEC_ERR_INVALID_ARG),
    (dict(head_dim=64), kvec.KVEC_ERR_UNSUPPORTED),
    (dict(obs_window=40), kvec.KVEC_ERR_INVALID_ARG),
    (dict(ext_window=0), kvec.KVEC_ERR_INVALID_ARG),
    (dict(pool_kernel=6), kvec.KVEC_ERR_INVALID_ARG),
    (dict(pool_kernel=17), kvec.KVEC_ERR_INVALID_ARG),
    (dict(num_ext_heads=9), kvec.KVEC_ERR_INVALID_ARG),
    (dict(beta=1.5), kvec.KVEC_ERR_INVALID_ARG),
    (dict(lam=float("inf")), kvec.KVEC_ERR_INVALID_ARG),
    (dict(max_layers=256), kvec.KVEC_ERR_INVALID_ARG),
    (dict(max_seqlen=0), kvec.KVEC_ERR_INVALID_ARG),
    (dict(max_seqlen=200000), kvec.KVEC_ERR_INVALID_ARG),
    (dict(num_q_heads=72, num_kv_heads=8), kvec.KVEC_ERR_UNSUPPORTED),   # 9 x 32 rows > 256
    (dict(num_q_heads=264, num_kv_heads=33), kvec.KVEC_ERR_UNSUPPORTED),
    (dict(all_positions=2), kvec.KVEC_ERR_INVALID_ARG),
    (dict(head_budget=2), kvec.KVEC_ERR_INVALID_ARG),
    (dict(head_budget=1, ada_floor=-0.1), kvec.KVEC_ERR_INVALID_ARG),
    (dict(head_budget=1, ada_floor=1.5), kvec.KVEC_ERR_INVALID_ARG),
    (dict(head_budget=1, ada_floor=float("nan")), kvec.KVEC_ERR_INVALID_ARG),
]


@pytest.mark.parametrize("over,code", BAD_PARAMS)
def test_create_rejects_bad_parameters_before_cuda(lib, over, code):
    kw = dict(num_q_heads=32, num_kv_heads=8)
    kw.update(over)
    p = kvec.make_params(**kw)
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_create(p)
    assert e.value.status == code
    assert kvec.load().kvec_last_error()


def test_calls_on_null_handle_are_rejected(lib):
    cu = (ctypes.c_int32 * 2)(0, 64)
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_select_layer(None, 1, ctypes.addressof(cu), ctypes.addressof(cu), 16, 16, 16, 16, 64, 16, 16, 16)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    for fn in (lambda: kvec.kvec_reset(None, 16, 1), lambda: kvec.kvec_sync_status(None),
               lambda: kvec.kvec_debug_scores(None), lambda: kvec.kvec_destroy(None)):
        with pytest.raises(kvec.KvecError):
            fn()


def test_status_strings(lib):
    for code in range(6):
        assert kvec.kvec_status_string(code)


@pytest.mark.parametrize("budget", [32, 33, 64, 128, 333, 2048])
@pytest.mark.parametrize("head_budget,ada_floor", [(0, 1.0), (1, 0.0), (1, 0.2), (1, 0.5), (1, 1.0)])
@pytest.mark.parametrize("all_positions", [0, 1])
def test_output_capacity_matches_oracle(lib, budget, head_budget, ada_floor, all_positions):
    p = kvec.make_params(num_q_heads=32, num_kv_heads=8, head_budget=head_budget, ada_floor=ada_floor,
                         all_positions=all_positions)
    op = oracle.OracleParams(num_q_heads=32, num_kv_heads=8, head_dim=128, window=p.window, obs_window=p.obs_window,
                             ext_window=p.ext_window, pool_kernel=p.pool_kernel, num_ext_heads=p.num_ext_heads,
                             beta=float(p.beta), lam=float(p.lam), head_criterion=p.head_criterion,
                             all_positions=all_positions, head_budget=head_budget, ada_floor=float(p.ada_floor))
    cap = kvec.kvec_output_capacity(p, budget)
    assert cap == oracle.head_capacity(op, budget)
    assert cap >= budget
    if head_budget == 0 or ada_floor == 1.0:
        assert cap == budget


def test_output_capacity_rejects_a_budget_below_the_window(lib):
    p = kvec.make_params(num_q_heads=32, num_kv_heads=8)
    with pytest.raises(kvec.KvecError):
        kvec.kvec_output_capacity(p, p.window - 1)


def test_noalloc_refuses_the_adaptive_fill_before_cuda(lib):
    p = kvec.make_params(num_q_heads=32, num_kv_heads=8, head_budget=1, ada_floor=0.2)
    cu = (ctypes.c_int32 * 2)(0, 4096)
    fake = 256
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_select_layer_noalloc(p, 1, ctypes.addressof(cu), ctypes.addressof(cu), fake, fake, fake, fake,
                                       512, fake, fake, fake, None)
    assert e.value.status == kvec.KVEC_ERR_UNSUPPORTED


def test_noalloc_refuses_oversize_calls_before_cuda(lib):
    # The scratch check comes before any CUDA call, so it runs without a GPU and the
    # (never dereferenced) pointers can be placeholders.
    batch, L = 16, 131072
    p = kvec.make_params(num_q_heads=32, num_kv_heads=8, max_batch=batch, max_seqlen=L)
    cu = (ctypes.c_int32 * (batch + 1))(*[b * L for b in range(batch + 1)])
    fake = 256
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_select_layer_noalloc(p, batch, ctypes.addressof(cu), ctypes.addressof(cu), fake, fake, fake, fake,
                                       512, fake, fake, fake, None)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    assert "scratch" in str(e.value)


@pytest.mark.parametrize("case,needle", [
    ("empty_batch", "batch 0"), ("batch_over_max", "batch 3"), ("cu_not_from_zero", "cu_seqlens[0]"),
    ("sequence_shorter_than_window", "length 31"), ("sequence_over_max_seqlen", "length 4097"),
    ("budget_below_window", "budget 31"), ("zero_budget", "budget 0"), ("null_k", "NULL"),
    ("misaligned_k", "aligned")])
def test_noalloc_validates_calls_before_cuda(lib, case, needle):
    # Degenerate and malformed calls: every one is refused by the host checks,
    # before any CUDA call (the placeholder pointers are never dereferenced).
    p = kvec.make_params(num_q_heads=32, num_kv_heads=8, max_batch=2, max_seqlen=4096)
    batch, budget, lens, first = 2, 256, [1000, 2000], 0
    fake = {n: 256 for n in ("q", "k", "v", "state", "out_idx", "out_k", "out_v")}
    if case == "empty_batch":
        batch = 0
    elif case == "batch_over_max":
        batch, lens = 3, [1000, 2000, 500]
    elif case == "cu_not_from_zero":
        first = 1
    elif case == "sequence_shorter_than_window":
        lens = [1000, p.window - 1]
    elif case == "sequence_over_max_seqlen":
        lens = [4097, 100]
    elif case == "budget_below_window":
        budget = p.window - 1
    elif case == "zero_budget":
        budget = 0
    elif case == "null_k":
        fake["k"] = 0
    elif case == "misaligned_k":
        fake["k"] = 256 + 2
    cu_vals = [first]
    for L in lens:
        cu_vals.append(cu_vals[-1] + L)
    cu = (ctypes.c_int32 * len(cu_vals))(*cu_vals)
    with pytest.raises(kvec.KvecError) as e:
        kvec.kvec_select_layer_noalloc(p, batch, ctypes.addressof(cu), ctypes.addressof(cu), fake["q"], fake["k"],
                                       fake["v"], fake["state"], budget, fake["out_idx"], fake["out_k"],
                                       fake["out_v"], None)
    assert e.value.status == kvec.KVEC_ERR_INVALID_ARG
    assert needle in str(e.value), str(e.value)


@pytest.mark.parametrize("struct", [kvec.kvec_params, kvec.kvec_debug_view])
def test_binding_structs_match_the_header_layout(tmp_path, struct):
    """Every field of the ctypes mirror sits at the offset (and the struct has the
    size) that a C compiler gives the declaration in include/kvec.h."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    name = struct.__name__
    c_name = {"lam": "lambda"}   # fields the binding renames (Python keywords)
    lines = [f'printf("size %zu\\n", sizeof({name}));']
    lines += [f'printf("{f} %zu\\n", offsetof({name}, {c_name.get(f, f)}));' for f, _ in struct._fields_]
    src = tmp_path / "layout.c"
    src.write_text("#include <stddef.h>\n#include <stdio.h>\n#include \"kvec.h\"\nint main(void) {\n" +
                   "\n".join(lines) + "\nreturn 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    out = dict(line.split() for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                        check=True).stdout.splitlines())
    assert int(out["size"]) == ctypes.sizeof(struct)
    for f, _ in struct._fields_:
        assert int(out[f]) == getattr(struct, f).offset, f
