"""Plant plausible mistakes in a copy of the oracle and check that the pins catch each.

The copy is compiled into a temporary directory; the committed oracle is never
modified.  A mutant that passes every pin would mean the pins leave that part
of the oracle unchecked.
"""
import os
import shutil
import subprocess

import pytest

import oracle
from tests import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "darb_oracle.c")

MUTANTS = {
    "tie_break_highest_index": ("> fabs(LOAD(W[r * ldw + best]))", ">= fabs(LOAD(W[r * ldw + best]))"),
    "floor_block_count": ("int64_t n = (cols + m[r] - 1) / m[r];", "int64_t n = cols / m[r];"),
    "keep_block_first_not_max": ("val[blk_ptr[r] + j] = W[r * ldw + best];",
                                 "val[blk_ptr[r] + j] = W[r * ldw + lo];"),
    "equal_density_rounds_down": ("} else if (nnz * rows >= total) {", "} else if (nnz * rows > total) {"),
    "round_up_off_by_one": ("while (2 * m * nnz <= cols) m *= 2;", "while (2 * m * nnz < cols) m *= 2;"),
    "round_down_off_by_one": ("while (m * nnz < cols) m *= 2;", "while (m * nnz <= cols) m *= 2;"),
    "product_wrong_sign": ("s += val[p] * X[k * ldx + b];", "s -= val[p] * X[k * ldx + b];"),
    "product_drops_offset": ("int64_t k = j * m[r] + off[p];\n                if (off[p] >= m[r] || k >= cols) { bad = 1; break; }",
                             "int64_t k = j * m[r];\n                if (off[p] >= m[r] || k >= cols) { bad = 1; break; }"),
    "product_drops_last_term": ("for (int64_t p = blk_ptr[r]; p < blk_ptr[r + 1]; ++p) {\n                int64_t j = p - blk_ptr[r];\n                int64_t k = j * m[r] + off[p];\n                if (off[p] >= m[r] || k >= cols) { bad = 1; break; }",
                                "for (int64_t p = blk_ptr[r]; p + 1 < blk_ptr[r + 1]; ++p) {\n                int64_t j = p - blk_ptr[r];\n                int64_t k = j * m[r] + off[p];\n                if (off[p] >= m[r] || k >= cols) { bad = 1; break; }"),
    "lstm_swaps_i_f": ("double c = sigmoid(gf) * c_prev[j * B + b] + sigmoid(gi) * tanh(gg);",
                       "double c = sigmoid(gi) * c_prev[j * B + b] + sigmoid(gf) * tanh(gg);"),
    "lstm_h_uses_old_c": ("h_out[j * B + b] = sigmoid(go) * tanh(c);",
                          "h_out[j * B + b] = sigmoid(go) * tanh(c_prev[j * B + b]);"),
    "lstm_drops_bias": ("double bb = bias ? bias[r] : 0.0;", "double bb = 0.0;"),
    "gru_reset_on_x_side": ("double nn = tanh(a[(2 * H + j) * B + b] + rr * bh[(2 * H + j) * B + b]);",
                            "double nn = tanh(rr * a[(2 * H + j) * B + b] + bh[(2 * H + j) * B + b]);"),
    "gru_swaps_z": ("h_out[j * B + b] = (1.0 - zz) * nn + zz * h_prev[j * B + b];",
                    "h_out[j * B + b] = zz * nn + (1.0 - zz) * h_prev[j * B + b];"),
    "gru_split_off_by_one": ("if (k < I) {", "if (k <= I) {"),
    "topk_strict_threshold": ("if (fabs(LOAD(W[r * ldw + c])) >= t) ++n;", "if (fabs(LOAD(W[r * ldw + c])) > t) ++n;"),
    "topk_off_by_one_rank": ("const double t = mag[keep - 1];", "const double t = mag[keep < rows * cols ? keep : keep - 1];"),
    "topk_ascending": ("return (x < y) - (x > y);", "return (x > y) - (x < y);"),
    "topk_signed_values": ("mag[r * cols + c] = fabs(v);", "mag[r * cols + c] = v;"),
}


def _build_mutant(tmp_path, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    path = tmp_path / f"{name}.c"
    path.write_text(src.replace(old, new))
    lib = tmp_path / f"lib{name}.so"
    cc = shutil.which("gcc") or shutil.which("cc")
    subprocess.run([cc, "-O1", "-std=c11", "-fPIC", "-shared", str(path), "-o", str(lib), "-lm"],
                   check=True, capture_output=True)
    return oracle.load_library(str(lib))


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(tmp_path, name):
    old, new = MUTANTS[name]
    mutant = _build_mutant(tmp_path, name, old, new)
    saved = oracle._load()
    caught = []
    try:
        oracle._lib = mutant
        for check in oracle_pins.ALL_CHECKS:
            try:
                check(oracle)
            except (AssertionError, oracle.OracleError):
                caught.append(check.__name__)
    finally:
        oracle._lib = saved
    assert caught, f"no pin caught mutant {name}"
