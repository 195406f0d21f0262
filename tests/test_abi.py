"""CPU checks of the boundary: libstill.so loads, exports every entry point include/still.h
declares, and its host-only accounting functions match the paper's printed numbers."""
import itertools
import json
import os
import re

import pytest

from paper_2606_07878_gb300 import still

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _declared():
    src = open(os.path.join(ROOT, "include", "still.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(still_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(still.LIB_PATH):
        from paper_2606_07878_gb300 import build
        build.build()
    return still.lib()


def test_exports_every_declared_symbol(lib):
    declared = _declared()
    assert declared, "no declarations parsed"
    assert sorted(still.EXPORTS) == declared
    for name in declared:
        assert hasattr(lib, name), name


def test_status_strings(lib):
    for code in still.STATUS:
        assert still.still_status_string(code)


def test_budget_matches_paper_table(lib):
    g = json.load(open(os.path.join(GOLDEN, "budgets.json")))
    for ctx, ratio, K in g["rows"]:
        assert still.still_budget(g["ctx_tokens"][ctx], ratio) == K


def test_kv_bytes_matches_paper(lib):
    g = json.load(open(os.path.join(GOLDEN, "kv_bytes.json")))
    m = g["model"]
    assert still.still_kv_bytes(m["L"], m["H"], m["d"], m["b"], 1) == 144 * 1024
    for S, gib in g["gib_at_tokens"]:
        assert still.still_kv_bytes(m["L"], m["H"], m["d"], m["b"], S) / 2**30 == pytest.approx(
            gib, abs=5e-4)


def test_param_count_matches_paper(lib):
    g = json.load(open(os.path.join(GOLDEN, "param_counts.json")))
    b = g["base"]
    for c in g["cases"]:
        cfg = still.make_config(b["H"], b["d"], c["D"], c["n"], c["r"] * c["D"], c["t"], 1e6,
                                n_blocks=c["B"], cross_every_block=int(c["cross_every_block"]))
        total = b["L"] * still.still_param_count(cfg, c["t"])
        assert abs(total - c["printed_total"]) <= g["tolerance_abs"], c["name"]


def test_lookahead_schedule_matches_oracle(lib):
    from oracle import still_oracle as O
    for k, c, t in itertools.product([0, 1, 2, 7, 127, 10**6], [1, 3, 8, 32], [1, 16, 128]):
        assert still.still_lookahead_pass_info(k, c, t) == O.lookahead_pass(k, c, t), (k, c, t)
    g = json.load(open(os.path.join(GOLDEN, "iterative_slots.json")))
    for case in g["cases"]:
        assert still.still_lookahead_totals(case["T"], case["c"], g["t"]) == O.lookahead_totals(
            case["T"], case["c"], g["t"])
    for args, name in [((1025, 8, 128), "STILL_ERR_SHAPE"), ((1024, 0, 128), "STILL_ERR_INVALID_ARG"),
                       ((0, 8, 128), "STILL_ERR_INVALID_ARG")]:
        with pytest.raises(still.StillError) as e:
            still.still_lookahead_totals(*args)
        assert e.value.name == name, args
    for args in [(-1, 8, 128), (0, 8, 0), (2**53, 8, 128)]:
        with pytest.raises(still.StillError) as e:
            still.still_lookahead_pass_info(*args)
        assert e.value.name == "STILL_ERR_INVALID_ARG", args


def test_new_entry_points_validate_on_the_host(lib):
    """Argument checks of the later entry points run before any device work (no GPU needed)."""
    import ctypes
    INVALID = 1
    assert lib.still_set_key_fold(None, 1) == INVALID
    assert lib.still_set_beta_head(None, 0, None, None, None) == INVALID
    assert lib.still_attend_biased(None, None, 1, 8, None, None, None, 0, None, None, 1, 8, 128,
                                   0.0, None, None) == INVALID
    mask = (ctypes.c_uint8 * 2)(1, 0)
    assert lib.still_compact_stack_masked(None, 2, mask, None, None, None, None, 0, 1, 1, None,
                                          None, None, None, None, None) == INVALID
    passes = (ctypes.c_int64 * 1)(0)
    assert lib.still_lookahead_compact_layer(None, 0, 1, None, None, passes, 8, 16, None, None,
                                             None) == INVALID
    assert lib.still_lookahead_compact_stack(None, 1, None, 1, None, None, passes, 8, 16, None,
                                             None, None) == INVALID
    # a negative pass index or a zero ratio is refused before the context is looked at
    bad = (ctypes.c_int64 * 1)(-1)
    assert lib.still_lookahead_compact_layer(None, 0, 1, None, None, bad, 8, 16, None, None,
                                             None) == INVALID
