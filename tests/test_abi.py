"""The C-ABI library loads without a GPU, exports exactly the entry points
include/dualmap.h declares, and the binding's struct layouts match the
header's as compiled by the host C compiler."""

import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HDR = os.path.join(ROOT, "include", "dualmap.h")


@pytest.fixture(scope="module")
def built():
    import __graft_entry__ as g
    g.build()
    from paper_2602_06502_gb300 import dualmap as D
    return D


def declared():
    txt = open(HDR).read()
    return sorted(set(re.findall(r"^DM_API [^(]*?\b(dm_\w+)\(", txt, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared()
    for must in ("dm_create", "dm_destroy", "dm_add_instance", "dm_remove_instance", "dm_route_batch",
                 "dm_commit_cache", "dm_rebalance"):
        assert must in names


def test_library_exports_every_declared_symbol(built):
    D = built
    exported = subprocess.run(["nm", "-D", "--defined-only", D.LIB_PATH], capture_output=True, text=True,
                              check=True).stdout
    syms = set(re.findall(r"\sT\s(dm_\w+)", exported))
    assert set(declared()) == syms
    assert set(D.SIGNATURES) == syms
    lib = C.CDLL(D.LIB_PATH)
    for s in declared():
        assert getattr(lib, s) is not None


def test_status_strings_without_gpu(built):
    D = built
    assert D.status_string(0) == "ok"
    assert "instances" in D.status_string(3)


def test_create_rejects_bad_config_without_touching_gpu(built):
    """Synchronous argument checks run before any CUDA call."""
    D = built

    def cfg(**kw):
        base = dict(block_tokens=16, route_prefix_blocks=16, vnodes_per_instance=8, max_instances=8,
                    cache_capacity_blocks=1024, slo_us=1, cost_us_per_token=1, hot_num=3, hot_den=2, max_batch=16,
                    max_batch_tokens=1 << 20, seed=1)
        base.update(kw)
        return D.dm_config(**base)

    h = C.c_void_p()
    for bad in (cfg(block_tokens=17), cfg(index_slots_log2=41), cfg(route_prefix_blocks=0),
                cfg(max_instances=1), cfg(choice_rule=D.DM_RULE_PREBLE + 1),
                cfg(adapt_step_blocks=4, adapt_max_blocks=16, adapt_window=1),    # cap not above K_route
                cfg(adapt_step_blocks=4, adapt_max_blocks=4096, adapt_window=1),  # cap above 2048
                cfg(adapt_step_blocks=4, adapt_max_blocks=64, adapt_window=0),
                cfg(rebalance_flags=4),
                cfg(rebuild_pool=1, index_slots_log2=12, max_touch_per_instance=1024)):   # 4 waits x 1024 > 2^11
        assert D.lib().dm_create(C.byref(bad), C.byref(h)) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_route_batch(None, None, None) == D.DM_ERR_INVALID_ARG


def test_potc_rejects_bad_arguments_without_touching_gpu(built):
    """dm_potc_max_loads checks its arguments before any CUDA call, and zero
    trials is a no-op."""
    D = built
    buf = C.c_void_p(16)   # never dereferenced: every call below returns before launching
    assert D.lib().dm_potc_max_loads(0, 10, 2, 4, 1, buf, None) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_potc_max_loads(257, 10, 2, 4, 1, buf, None) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_potc_max_loads(8, 10, 0, 4, 1, buf, None) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_potc_max_loads(8, 10, 65, 4, 1, buf, None) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_potc_max_loads(8, 1 << 32, 2, 4, 1, buf, None) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_potc_max_loads(8, 10, 2, 4, 1, None, None) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_potc_max_loads(8, 10, 2, 0, 1, buf, None) == D.DM_OK


def test_read_back_calls_reject_a_null_handle_without_touching_gpu(built):
    D = built
    m = D.dm_metrics()
    n = C.c_uint64()
    assert D.lib().dm_get_metrics(None, C.byref(m), None, 0, 0) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_export_prefix_tree(None, None, 0, C.byref(n)) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_get_route_blocks(None, None, 0) == D.DM_ERR_INVALID_ARG


def test_struct_layouts_match_header(built, tmp_path):
    D = built
    prog = tmp_path / "layout.c"
    fields = {
        "dm_config": [f for f, _ in D.dm_config._fields_],
        "dm_batch": [f for f, _ in D.dm_batch._fields_],
        "dm_route_out": [f for f, _ in D.dm_route_out._fields_],
        "dm_route_out_d": [f for f, _ in D.dm_route_out_d._fields_],
        "dm_migration": ["req_seq", "from", "to"],
        "dm_metrics": [f for f, _ in D.dm_metrics._fields_],
    }
    lines = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HDR}"', "int main(void) {"]
    for st, fs in fields.items():
        lines.append(f'printf("{st} %zu\\n", sizeof({st}));')
        for f in fs:
            lines.append(f'printf("{st}.{f} %zu\\n", offsetof({st}, {f}));')
    consts = ["DM_HIST_BUCKETS", "DM_REBALANCE_SLO_TARGET", "DM_REBALANCE_DOUBLE_OVERLOAD"] + \
        [f"DM_RULE_{n.upper()}" for n in D.RULE_NAMES]
    for c in consts:
        lines.append(f'printf("{c} %u\\n", (unsigned){c});')
    lines.append("return 0; }")
    prog.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", str(prog), "-o", str(exe)], check=True)
    out = dict(l.rsplit(" ", 1) for l in subprocess.run([str(exe)], capture_output=True, text=True,
                                                        check=True).stdout.split("\n") if l)
    for c in consts:
        assert int(out[c]) == getattr(D, c), c
    for st, cls in (("dm_config", D.dm_config), ("dm_batch", D.dm_batch), ("dm_route_out", D.dm_route_out),
                    ("dm_route_out_d", D.dm_route_out_d),
                    ("dm_migration", D.dm_migration), ("dm_metrics", D.dm_metrics)):
        assert int(out[st]) == C.sizeof(cls), st
        for (py, _), cn in zip(cls._fields_, fields[st]):
            assert int(out[f"{st}.{cn}"]) == getattr(cls, py).offset, (st, cn)


def test_boundary_signatures_compile_against_the_scope_table(tmp_path):
    """The calls of the routing boundary keep the signatures of the
    hot-path scope table (dm_rebalance and dm_get_loads with host results
    and a count): a C program that binds each to a pointer of exactly that
    type compiles with incompatible-pointer warnings as errors."""
    prog = tmp_path / "sig.c"
    prog.write_text("\n".join([
        f'#include "{HDR}"',
        "dm_status (*p_create)(const dm_config *, dm_handle **) = dm_create;",
        "void (*p_destroy)(dm_handle *) = dm_destroy;",
        "dm_status (*p_add)(dm_handle *, uint32_t) = dm_add_instance;",
        "dm_status (*p_remove)(dm_handle *, uint32_t) = dm_remove_instance;",
        "dm_status (*p_route)(dm_handle *, const dm_batch *, const dm_route_out *) = dm_route_batch;",
        "dm_status (*p_commit)(dm_handle *) = dm_commit_cache;",
        "dm_status (*p_rebalance)(dm_handle *, dm_migration *, uint32_t, uint32_t *) = dm_rebalance;",
        "dm_status (*p_loads)(dm_handle *, uint64_t *, uint32_t, uint32_t *) = dm_get_loads;",
        "dm_status (*p_err)(dm_handle *) = dm_last_error;",
        "int main(void) { return 0; }",
    ]))
    subprocess.run(["gcc", "-c", "-Werror", "-Wincompatible-pointer-types", str(prog), "-o",
                    str(tmp_path / "sig.o")], check=True)


def test_host_result_calls_check_arguments_without_touching_gpu(built):
    D = built
    n = C.c_uint32()
    w = (C.c_uint64 * 4)()
    mig = (D.dm_migration * 4)()
    assert D.lib().dm_get_loads(None, w, 4, C.byref(n)) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_rebalance(None, mig, 4, C.byref(n)) == D.DM_ERR_INVALID_ARG
    assert D.lib().dm_rebalance_async(None, None, 0, None) == D.DM_ERR_INVALID_ARG


def test_allocation_failure_hook_gives_oom_without_a_gpu(built):
    """dm_test_fail_alloc(0) fails dm_create's first device allocation
    before any CUDA allocator call: DM_ERR_OOM and no handle, on the CPU;
    out-of-range candidate counts are refused before any allocation."""
    D = built
    cfg = D.dm_config(block_tokens=16, route_prefix_blocks=16, vnodes_per_instance=8, max_instances=8,
                      cache_capacity_blocks=1024, slo_us=1, cost_us_per_token=1, hot_num=3, hot_den=2, max_batch=16,
                      max_batch_tokens=1 << 20, seed=1)
    h = C.c_void_p()
    D.lib().dm_test_fail_alloc(0)
    try:
        assert D.lib().dm_create(C.byref(cfg), C.byref(h)) == D.DM_ERR_OOM
        assert not h.value
    finally:
        D.lib().dm_test_fail_alloc(-1)
    bad = D.dm_config(block_tokens=16, route_prefix_blocks=16, vnodes_per_instance=8, max_instances=8,
                      cache_capacity_blocks=1024, slo_us=1, cost_us_per_token=1, hot_num=3, hot_den=2, max_batch=16,
                      max_batch_tokens=1 << 20, seed=1, candidates=9)
    assert D.lib().dm_create(C.byref(bad), C.byref(h)) == D.DM_ERR_INVALID_ARG
    bad.candidates, bad.choice_rule = 3, D.DM_RULE_PAIR_MIN_TTFT   # the d-way path takes DualMap's rule only
    assert D.lib().dm_create(C.byref(bad), C.byref(h)) == D.DM_ERR_INVALID_ARG
