"""The pins catch plausible mistakes in the oracle.

Each case plants one mistake (a dropped term, a wrong sign, a transposed
operand, an off-by-one comparison, a missing reset) into a copy of the C
oracle, builds it on the CPU, and runs the listed pins against it in a
child process; at least one pin must fail (an assertion, or a crash the
mistake causes).  No GPU is involved."""
import os
import subprocess
import sys
import tempfile

import pytest

from tests.conftest import ROOT

SRC = os.path.join(ROOT, "oracle", "lc_oracle.c")

MUTATIONS = [
    ("abs-of-difference-split", "d_sum += fabs(w - r);", "d_sum += fabs(w) - fabs(r);",
     ["test_sums_depend_on_reference_not_current_for_denominator", "test_measure_hand_cases"]),
    ("difference-sign", "d_sum += fabs(w - r);", "d_sum += fabs(w + r);",
     ["test_measure_hand_cases", "test_unchanged_layer_measures_zero"]),
    ("denominator-uses-current", "a_sum += fabs(r);", "a_sum += fabs(w);",
     ["test_measure_hand_cases", "test_sums_depend_on_reference_not_current_for_denominator"]),
    ("epsilon-dropped", "mean_abs_update / (mean_abs_weight + eps_w)",
     "mean_abs_update / (mean_abs_weight)", ["test_measure_hand_cases"]),
    ("mean-over-first-tensor-count", "n += t[k].numel;", "if (k == 0) n += t[k].numel;",
     ["test_measure_hand_cases"]),
    ("bf16-shift", "((uint32_t)bits) << 16", "((uint32_t)bits) << 15",
     ["test_bf16_value_known_patterns"]),
    ("strict-threshold", "acc >= threshold", "acc > threshold",
     ["test_select_golden_sequences", "test_threshold_tie_and_epsilon_h1"]),
    ("strict-staleness", "staleness >= (int64_t)max_staleness", "staleness > (int64_t)max_staleness",
     ["test_select_golden_sequences", "test_table1_default_layer_writes"]),
    ("no-reset-on-persist", "delta[l] = 0.0;", "delta[l] = acc;",
     ["test_select_golden_sequences", "test_select_brute_force_against_history_rule"]),
    ("snapshot-accumulates", "(mode == LCO_ACCUMULATE) ? delta[l] + u[l] : u[l]", "delta[l] + u[l]",
     ["test_select_golden_sequences"]),
    ("no-nonfinite-guard", "if (!isfinite(acc)) {", "if (0) {", ["test_select_golden_sequences"]),
    ("t_last-not-updated", "t_last[l] = t;", "(void)t;",
     ["test_select_golden_sequences", "test_staleness_bound_holds_over_random_runs"]),
    ("threshold-ignores-multiplier", "tau * (tau_mult ? tau_mult[l] : 1.0)", "tau",
     ["test_tau_multiplier_embedding_threshold"]),
    ("staleness-weights-dropped", "num += (double)layer_numel[l] * (double)s;", "num += (double)s;",
     ["test_staleness_closed_form"]),
    ("moments-before-weights", "const void* src = part == 0 ? t[k].w : part == 1",
     "const void* src = part == 1 ? t[k].w : part == 0", ["test_pack_layout_by_independent_parse"]),
    ("padding-not-zeroed", "memset(dst + off + sz[part], 0, padded - sz[part]);",
     "memset(dst + off + sz[part], 0x5A, padded - sz[part]);", ["test_pack_layout_by_independent_parse"]),
    ("composite-off-by-one", "v_step[i] > t_fail", "v_step[i] >= t_fail",
     ["test_composite_pick_equals_replay"]),
    ("composite-ignores-durability", "!v_durable[i] ||", "",
     ["test_composite_pick_equals_replay", "test_crash_before_durable_uses_previous_version"]),
    ("composite-first-not-latest", "v_step[i] >= v_step[pick_out[l]]", "0",
     ["test_composite_pick_equals_replay", "test_composite_equals_latest_persisted_versions"]),
    ("adamw-no-second-bias-correction", "const float v_hat = v_new * rbc2;", "const float v_hat = v_new;",
     ["test_adamw_hand_cases", "test_constant_gradient_closed_form"]),
    ("adamw-no-first-bias-correction", "out[5] = (float)(hp->lr / (1.0 - pow(hp->beta1, (double)t)));",
     "out[5] = (float)hp->lr;", ["test_adamw_hand_cases", "test_constant_gradient_closed_form"]),
    ("adamw-second-moment-linear", "const float gg = g * g;", "const float gg = g;",
     ["test_adamw_hand_cases", "test_matches_binary64_adamw_within_fp32_rounding"]),
    ("adamw-decay-dropped", "const float p_decayed = p_old * decay;", "const float p_decayed = p_old;",
     ["test_adamw_hand_cases"]),
    ("adamw-drift-against-decayed", "d_sum += fabs((double)p_new - (double)p_old);",
     "d_sum += fabs((double)p_new - (double)p_decayed);",
     ["test_adamw_hand_cases", "test_fused_drift_sums_are_eq1_of_the_update"]),
    ("bf16-round-truncates", "return (uint16_t)((u + 0x7fffu + keep_lsb) >> 16);",
     "return (uint16_t)(u >> 16); (void)keep_lsb;", ["test_fused_drift_sums_are_eq1_of_the_update",
                                                      "test_bf16_round_matches_torch"]),
]

RUNNER = r"""
import ctypes, sys
sys.path.insert(0, sys.argv[1])
from oracle import oracle as O
O._lib = O.declare(ctypes.CDLL(sys.argv[2]))
from tests import test_oracle_pins as pins, test_oracle_adamw as pins_adamw
failed = []
for name in sys.argv[3:]:
    fn = pins.__dict__.get(name) or pins_adamw.__dict__[name]
    args = fn.__code__.co_varnames[:fn.__code__.co_argcount]
    kw = {k: v for k, v in (("oracle_lib", None), ("align", 256), ("dtype", "bf16")) if k in args}
    try:
        fn(**kw)
    except Exception as e:
        failed.append(name)
print("FAILED:" + ",".join(failed))
sys.exit(3 if failed else 0)
"""


def _build_mutant(old, new, tmp):
    text = open(SRC).read()
    assert text.count(old) == 1, "mutation anchor must occur exactly once: %r" % old
    src = os.path.join(tmp, "lc_oracle.c")
    open(src, "w").write(text.replace(old, new))
    lib = os.path.join(tmp, "libmut.so")
    subprocess.run(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-w",
                    "-I", os.path.join(ROOT, "oracle"), "-o", lib, src, "-lm"], check=True)
    return lib


@pytest.mark.parametrize("name,old,new,tests", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_planted_mistake(name, old, new, tests):
    with tempfile.TemporaryDirectory() as tmp:
        lib = _build_mutant(old, new, tmp)
        r = subprocess.run([sys.executable, "-c", RUNNER, ROOT, lib, *tests],
                           capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, "mutation %s passed every pin in %s\n%s" % (name, tests, r.stdout)


def test_genuine_oracle_passes_the_same_runner():
    from oracle.build import build_oracle
    names = sorted({t for m in MUTATIONS for t in m[3]})
    r = subprocess.run([sys.executable, "-c", RUNNER, ROOT, build_oracle(), *names],
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr


# ----------------------------------------------------------------------------
# the file-tier oracle (oracle/files.py): the same idea for its Python form
# ----------------------------------------------------------------------------
FILES_SRC = os.path.join(ROOT, "oracle", "files.py")

FILES_MUTATIONS = [
    ("crc-polynomial-term-dropped", "(0, 6, 8, 9, 10, 11, 13, 14, 18, 19, 20, 22, 23, 25, 26, 27, 28)",
     "(0, 6, 8, 9, 10, 11, 13, 14, 18, 19, 20, 22, 23, 25, 26, 27)", ["test_crc32c_check_value_and_forms"]),
    ("crc-no-final-inversion", "reg = (reg >> 8) ^ t[(reg ^ byte) & 0xFF]\n    return reg ^ 0xFFFFFFFF",
     "reg = (reg >> 8) ^ t[(reg ^ byte) & 0xFF]\n    return reg", ["test_crc32c_check_value_and_forms"]),
    ("crc-table-index-drops-register", "t[(reg ^ byte) & 0xFF]", "t[byte & 0xFF]",
     ["test_crc32c_check_value_and_forms"]),
    ("pick-tie-keeps-first-record", 'r["step"] >= recs[best[l]]["step"]', 'r["step"] > recs[best[l]]["step"]',
     ["test_pick_matches_composite_rule_and_replay"]),
    ("pick-past-t_fail", 'r["step"] > t_fail', 'r["step"] > t_fail + 1',
     ["test_pick_matches_composite_rule_and_replay"]),
    ("pick-ignores-damage", ' or not r.get("intact", True)', "",
     ["test_pick_matches_composite_rule_and_replay", "test_damaged_block_is_not_intact"]),
    ("pick-ignores-block-size", 'r["bytes"] != layer_bytes[l] or ', "",
     ["test_pick_matches_composite_rule_and_replay"]),
    ("reader-skips-a-bad-record", "            break\n        layer, step",
     "            off += REC\n            continue\n        layer, step", ["test_torn_tail_and_damaged_record_end_the_log"]),
    ("record-offset-and-size-swapped", 'pack("<iqQQII", layer, step, offset, nbytes, block_crc, layout)',
     'pack("<iqQQII", layer, step, nbytes, offset, block_crc, layout)',
     ["test_manifest_read_matches_independent_writer"]),
    ("verify-ignores-block-crc", 'len(blk) == r["bytes"] and crc_of(blk) == r["block_crc"]', 'len(blk) == r["bytes"]',
     ["test_damaged_block_is_not_intact"]),
]

RUNNER_FILES = r"""
import importlib.util, pathlib, sys, tempfile
sys.path.insert(0, sys.argv[1])
import oracle
spec = importlib.util.spec_from_file_location("oracle.files", sys.argv[2])
mod = importlib.util.module_from_spec(spec)
sys.modules["oracle.files"] = mod
spec.loader.exec_module(mod)
oracle.files = mod
from tests import test_files as T
P = None
failed = []
for name in sys.argv[3:]:
    fn = T.__dict__[name]
    args = fn.__code__.co_varnames[:fn.__code__.co_argcount]
    kw = {}
    if "P" in args:
        if P is None:
            from paper_2609_27193_gb300 import build as B
            B.build()
            import paper_2609_27193_gb300 as P
        kw["P"] = P
    with tempfile.TemporaryDirectory() as d:
        if "tmp_path" in args:
            kw["tmp_path"] = pathlib.Path(d)
        try:
            fn(**kw)
        except Exception:
            failed.append(name)
print("FAILED:" + ",".join(failed))
sys.exit(3 if failed else 0)
"""


def _files_mutant(old, new, tmp):
    text = open(FILES_SRC).read()
    assert text.count(old) == 1, "mutation anchor must occur exactly once: %r" % old
    path = os.path.join(tmp, "files.py")
    open(path, "w").write(text.replace(old, new))
    return path


@pytest.mark.parametrize("name,old,new,tests", FILES_MUTATIONS, ids=[m[0] for m in FILES_MUTATIONS])
def test_file_tier_pins_catch_planted_mistake(name, old, new, tests):
    with tempfile.TemporaryDirectory() as tmp:
        path = _files_mutant(old, new, tmp)
        r = subprocess.run([sys.executable, "-c", RUNNER_FILES, ROOT, path, *tests],
                           capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, "mutation %s passed every pin in %s\n%s%s" % (name, tests, r.stdout, r.stderr)


def test_genuine_file_tier_oracle_passes_the_same_runner():
    names = sorted({t for m in FILES_MUTATIONS for t in m[3]})
    r = subprocess.run([sys.executable, "-c", RUNNER_FILES, ROOT, FILES_SRC, *names],
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
