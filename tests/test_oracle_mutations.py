"""The oracle's pins must catch plausible mistakes.

Each case copies oracle.c, plants one mistake (a dropped term, a wrong index,
a swapped operand), builds the copy on the CPU and runs the pin suite against
it in a subprocess: the suite must fail.  The committed oracle is untouched.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.c")

MUTANTS = {
    "no_live_check": ("if (!p->live[s]) return 0;", "if (0) return 0;"),
    "eos_ignores_stack": ("return p->accepting[s] && st->depth == 0;", "return p->accepting[s];"),
    "pop_ignores_top": ("st->sym[st->depth - 1] != p->rules[r].sym) return 0;", "0) return 0;"),
    "push_ignores_bound": ("if (st->depth == p->max_depth) return 0;", "if (0) return 0;"),
    "revealed_swapped": ("else if (st->sym[st->depth - 1] == 0) s = p->rules[r].next_if_top0;",
                         "else if (st->sym[st->depth - 1] == 1) s = p->rules[r].next_if_top0;"),
    "ties_highest_index": ("if (x > m) { m = x; best = t; }", "if (x >= m) { m = x; best = t; }"),
    "lse_drops_max": ("l = m + log(sum);", "l = log(sum);"),
    "mask_bit_shifted": ("mrow[t / 32] |= 1u << (t % 32);", "mrow[t / 32] |= 1u << ((t + 1) % 32);"),
    "empty_token_allowed": ("if (hi == lo) return 0;", "if (0) return 0;"),
    "bf16_wrong_shift": ("((const uint16_t*)logits)[i] << 16;", "((const uint16_t*)logits)[i] << 15;"),
    "stack_top_at_wrong_end": ("(uint8_t)((bits >> (st->depth - 1 - i)) & 1);", "(uint8_t)((bits >> i) & 1);"),
    "advance_eos_keeps_state": ("s_out = start_state;", "s_out = s;"),
    "gumbel_sign_flipped": ("float g = -oracle_ln_f32(e1);", "float g = oracle_ln_f32(e1);"),
    "temperature_multiplies": ("const float inv_t = 1.0f / temperature;", "const float inv_t = temperature;"),
    "philox_word_ignores_token": ("uint32_t k = c[t % 4] >> 9;", "uint32_t k = c[0] >> 9;"),
    "philox_rounds_short": ("for (int round = 0; round < 10; round++) {", "for (int round = 0; round < 9; round++) {"),
    "ln_series_term_dropped": ("poly = fmaf(poly, z2, 0x1.99999ap-3f);           /* 1/5 */", "poly = poly;"),
    "spec_ties_highest_id": ("sp->tok[key][i] < best)) {", "sp->tok[key][i] > best)) {"),
    "spec_threshold_strict": ("best_c * 1000 < (int64_t)min_permille * reached) break;",
                              "best_c * 1000 <= (int64_t)min_permille * reached) break;"),
    "spec_key_ignores_top": ("return state * 3 + top;", "return state * 3;"),
    "spec_chain_not_advanced": ("            state = end;\n            st = next;", "            st = next;"),
}
PIN_FILES = ["test_oracle_pins.py", "test_oracle_sampling.py", "test_oracle_spec.py"]


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(tmp_path, name):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, name
    d = tmp_path / "oracle"
    d.mkdir()
    shutil.copy(os.path.join(ROOT, "oracle", "oracle.h"), d / "oracle.h")
    (d / "oracle.c").write_text(src.replace(old, new))
    so = d / "liboracle_mutant.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", str(so), str(d / "oracle.c"),
                    "-lm"], check=True)
    env = dict(os.environ, DOMINO_ORACLE_SO=str(so))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        *[os.path.join(ROOT, "tests", f) for f in PIN_FILES]],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"mutant {name} survived the pins:\n{r.stdout[-2000:]}"
