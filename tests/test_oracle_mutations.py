"""Plant plausible mistakes in copies of the CPU oracle and check that the pins
catch every one of them (the planted copies live in a temporary directory)."""
import os
import shutil
import subprocess

import pytest

from oracle import oracle as O
from tests import _pins

SRC = os.path.join(os.path.dirname(O.__file__), "gba_oracle.c")

# (name, original text, planted text, occurrence index to replace)
MUTATIONS = [
    ("decay-boundary-strict", "if (s > (int64_t)rule->iota) return 0.0f;",
     "if (s >= (int64_t)rule->iota) return 0.0f;", 0),
    ("dense-divides-by-kept", "float g = gsum / (float)M;",
     "float g = gsum / (float)(st.msgs_kept > 0 ? st.msgs_kept : 1);", 0),
    ("row-divides-by-kept-messages", "int64_t denom = cnt[r];", "int64_t denom = cnt_kept[r];", 0),
    ("row-uses-message-staleness", "int64_t ref = (rule->row_staleness == 0) ? tb->ver[r] : k;",
     "int64_t ref = k;", 0),
    ("tag-not-compared", "int64_t ref = (rule->row_staleness == 0) ? tb->ver[r] : k;",
     "int64_t ref = tokens[m];", 0),
    ("adagrad-sign", "*w = *w - step / den;", "*w = *w + step / den;", 0),
    ("adagrad-old-accumulator", "float den = sqrtf(an);", "float den = sqrtf(*a);", 0),
    ("row-transposed", "S[r * d + j] += (double)fo * (double)gm[i * d + j];",
     "S[r * d + j] += (double)fo * (double)gm[j * nm + i];", 0),
    ("no-skip-of-dropped-rows", "if (kept_occ[r] == 0) continue;", "if (kept_occ[r] < 0) continue;", 0),
    ("adam-step-count", "int64_t t_step = k + 1;", "int64_t t_step = k + 2;", 0),
    ("counts-occurrences", "if (last_m[r] != m) {", "if (1) {", 0),
    ("adam-moment-order", "float mn = o->beta1 * *m + c1 * g;", "float mn = c1 * *m + o->beta1 * g;", 0),
    ("dense-drop-ignored", "if (f[m] > 0.0f) S += (double)f[m] * (double)dense_grads[m][e];",
     "S += (double)dense_grads[m][e];", 0),
    ("init-scale", "return (float)top * 0x1p-27f;", "return (float)top * 0x1p-26f;", 0),
    ("fifo-overshoot", "if (acc >= G) return i + 1;", "if (acc > G) return i + 1;", 0),
    # the optional readings (kept-message and M denominators, message staleness for rows)
    ("kept-denominator-counts-all", "if (rule->sparse_denominator == 1) denom = cnt_kept[r];",
     "if (rule->sparse_denominator == 1) denom = cnt[r];", 0),
    ("kept-denominator-counts-occurrences", "if (rule->sparse_denominator == 1) denom = cnt_kept[r];",
     "if (rule->sparse_denominator == 1) denom = kept_occ[r];", 0),
    ("m-denominator-counts-all", "if (rule->sparse_denominator == 2) denom = M;",
     "if (rule->sparse_denominator == 2) denom = cnt[r];", 0),
    ("m-denominator-counts-kept", "if (rule->sparse_denominator == 2) denom = M;",
     "if (rule->sparse_denominator == 2) denom = st.msgs_kept;", 0),
    ("message-staleness-option-ignored", "int64_t ref = (rule->row_staleness == 0) ? tb->ver[r] : k;",
     "int64_t ref = tb->ver[r];", 0),
    ("message-staleness-off-by-one", "int64_t ref = (rule->row_staleness == 0) ? tb->ver[r] : k;",
     "int64_t ref = (rule->row_staleness == 0) ? tb->ver[r] : k + 1;", 0),
    # decay strategies and Hop-BW
    ("geometric-exponent-off-by-one", "for (int64_t i = 0; i < s; ++i) p = p * (double)rule->lambda;",
     "for (int64_t i = 0; i <= s; ++i) p = p * (double)rule->lambda;", 0),
    ("geometric-ignored", "if (rule->decay == 0) return 1.0f;", "if (rule->decay >= 0) return 1.0f;", 0),
    ("row-weight-not-applied", "S[r * d + j] += (double)fo * (double)gm[i * d + j];",
     "S[r * d + j] += (double)gm[i * d + j];", 0),
    ("dense-weight-not-applied", "if (f[m] > 0.0f) S += (double)f[m] * (double)dense_grads[m][e];",
     "if (f[m] > 0.0f) S += (double)dense_grads[m][e];", 0),
    ("hopbw-drops-earliest", "if (m >= M - rule->drop_latest) return 0.0f;",
     "if (m < rule->drop_latest) return 0.0f;", 0),
    ("hopbw-off-by-one", "if (m >= M - rule->drop_latest) return 0.0f;",
     "if (m > M - rule->drop_latest) return 0.0f;", 0),
    ("hash-reserved-id-accepted", "if (id == INT64_MIN) { err = 1; continue; }",
     "if (id == INT64_MIN) { x = id; }", 0),
    ("adam-eps-inside-sqrt", "float den = sqrtf(vhat) + o->eps;", "float den = sqrtf(vhat + o->eps);", 0),
    ("adam-no-bias-correction", "float mhat = mn / bc1;", "float mhat = mn;", 0),
    ("tag-set-to-k", "tb->ver[r] = k + 1;", "tb->ver[r] = k;", 0),
    ("staleness-not-clamped", "return s < 0 ? 0 : s;", "return s;", 0),
    ("adagrad-init-zero", "tb->s0[i] = tb->opt.init_acc;", "tb->s0[i] = 0.0f;", 0),
    ("modulo-signed-residue", "x = (int64_t)((uint64_t)id % (uint64_t)tb->V);",
     "x = id % tb->V; if (x < 0) x += tb->V;", 0),
    ("hash-ids-folded", "  /* the reserved id */\n          x = id;",
     "  /* the reserved id */\n          x = (int64_t)((uint64_t)id % (uint64_t)tb->V);", 0),
]


def _plant(tmp_path, name, old, new, occ):
    src = open(SRC).read()
    idx = -1
    for _ in range(occ + 1):
        idx = src.index(old, idx + 1)
    planted = src[:idx] + new + src[idx + len(old):]
    c = tmp_path / f"{name}.c"
    so = tmp_path / f"{name}.so"
    c.write_text(planted)
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-shared", "-fPIC",
                           "-o", str(so), str(c), "-lm"])
    return O.load(str(so))


@pytest.mark.parametrize("mut", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_planted_mistake(tmp_path, mut):
    if shutil.which("gcc") is None:
        pytest.skip("gcc missing")
    L = _plant(tmp_path, *mut)
    caught = []
    for pin in _pins.ALL_PINS + [_pins.pin_init_published]:
        try:
            pin(L)
        except (AssertionError, ValueError, FloatingPointError):
            caught.append(pin.__name__)
    assert caught, f"no pin caught the planted mistake {mut[0]}"
