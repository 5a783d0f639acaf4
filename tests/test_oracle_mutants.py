"""Plant plausible mistakes in copies of the oracle and check that the pins catch each one.

Every mutant is a one-token edit of ``oracle/wino_oracle.c`` (a dropped term,
a flipped sign or comparison, a wrong index, a transposed row kind, a lost
rule), compiled on the CPU into a temporary library and run through the
pins of ``oracle_pins`` in a child process; at least one pin must fail (or
the mutant crash) for every mutant.
"""
import shutil
import subprocess
import sys
from pathlib import Path

import pytest

import oracle

SRC = Path(oracle.__file__).resolve().parent / "wino_oracle.c"

# (name, text in the oracle, replacement)
MUTANTS = [
    ("draft_not_strict", "(pmax[row_blk + l] > tau1)", "(pmax[row_blk + l] >= tau1)"),
    ("verify_not_strict", "(ptarget[row_shd + l] < tau2)", "(ptarget[row_shd + l] <= tau2)"),
    ("draft_reads_shadow_row", "(pmax[row_blk + l] > tau1)", "(pmax[row_shd + l] > tau1)"),
    ("verify_reads_block_row", "(ptarget[row_shd + l] < tau2)", "(ptarget[row_blk + l] < tau2)"),
    ("draft_ignores_mask_state", "(draft_m <= 0) && (prev[l] == mask_id) && ", "(draft_m <= 0) && "),
    ("verify_ignores_mask_state", "inR[l] = !no_shadow && (prev[l] != mask_id) && ", "inR[l] = !no_shadow && "),
    ("verify_runs_without_shadow", "inR[l] = !no_shadow && ", "inR[l] = "),
    ("no_fallback", "if (n_draft == 0 && n_mask > 0) {", "if (0) {"),
    ("fallback_last_on_ties", "pmax[row_blk + l] > best)) {", "pmax[row_blk + l] >= best)) {"),
    ("fallback_ignores_mask_state", "if (prev[l] == mask_id && (fallback < 0", "if ((fallback < 0"),
    ("argmax_last_on_ties", "if (logit[v] > m) {", "if (logit[v] >= m) {"),
    ("softmax_drops_term", "for (int64_t v = 0; v < V; ++v)\n                Z += exp",
     "for (int64_t v = 1; v < V; ++v)\n                Z += exp"),
    ("softmax_sign_flip", "Z += exp(logit[v] - m);", "Z += exp(m - logit[v]);"),
    ("pmax_not_inverted", "pmax[n] = 1.0 / Z;", "pmax[n] = Z / V;"),
    ("ptarget_uses_argmax", "exp(logit[t] - m) / Z", "exp(logit[a] - m) / Z"),
    ("hidden_index_reversed", "hd[k] = oracle_bf16_to_double(h[k]);", "hd[k] = oracle_bf16_to_double(h[d - 1 - k]);"),
    ("weight_row_stride_wrong", "const uint16_t *w = W + v * d;", "const uint16_t *w = W + v;"),
    ("bf16_wrong_shift", "(uint32_t)bits << 16;", "(uint32_t)bits << 15;"),
    ("verify_target_on_block_row", "target[(s * 2 + 1) * blk_len + l] = (y == mask_id) ? -1 : y;",
     "target[(s * 2 + 0) * blk_len + l] = (y == mask_id) ? -1 : y;"),
    ("remask_not_counted", "++remasked;", ""),
    ("left_counts_old_state", "left += (y[l] == mask_id);", "left += (prev[l] == mask_id);"),
    ("entropy_sign_flip", "h -= p * log(p);", "h += p * log(p);"),
    ("entropy_unnormalised", "const double p = exp(logit[v] - m) / Z;", "const double p = exp(logit[v] - m);"),
    ("freeze_ignored", "if (freeze_finished && n_mask == 0) {", "if (0) {"),
    ("freeze_always", "if (freeze_finished && n_mask == 0) {", "if (n_mask == 0) {"),
    ("last_change_on_every_position", "if (last_change && y[l] != before)", "if (last_change)"),
    ("fixed_m_last_on_ties", "pmax[row_blk + l] > pmax[row_blk + pick]", "pmax[row_blk + l] >= pmax[row_blk + pick]"),
    ("fixed_m_one_extra", "j < draft_m && j < n_mask", "j <= draft_m && j < n_mask"),
    ("fixed_m_keeps_threshold", "inD[l] = (draft_m <= 0) && ", "inD[l] = "),
    ("fixed_m_ignores_mask_state", "if (prev[l] == mask_id && !inD[l] && ", "if (!inD[l] && "),
    ("last_change_off_by_one", "last_change[s * seq_len + blk_start + l] = step_index;",
     "last_change[s * seq_len + blk_start + l] = step_index - 1;"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_kill_mutant(tmp_path, name, old, new):
    src = SRC.read_text()
    assert src.count(old) >= 1, f"mutation site for {name} not found"
    mutated = src.replace(old, new, 1)
    c = tmp_path / "mutant.c"
    c.write_text(mutated)
    so = tmp_path / f"liboracle_{name}.so"
    gcc = shutil.which("gcc")
    assert gcc
    r = subprocess.run([gcc, "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-fopenmp", str(c),
                        "-o", str(so), "-lm"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    # Run the pins on the mutant in a child process: a mutant may also crash (e.g. read through a
    # pointer the real oracle never touches in that mode), which counts as caught.
    here = Path(__file__).resolve().parent
    code = ("import sys; sys.path[:0] = [%r, %r]\n"
            "import oracle\nfrom oracle_pins import ALL_PINS\n"
            "O = oracle.Oracle(%r)\n"
            "for pin in ALL_PINS:\n"
            "    try:\n        pin(O)\n"
            "    except AssertionError:\n        print('caught by', pin.__name__); sys.exit(3)\n"
            "print('survived'); sys.exit(0)\n") % (str(here.parent), str(here), str(so))
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"no pin caught mutant {name}: {r.stdout}{r.stderr[-2000:]}"
