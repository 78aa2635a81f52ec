"""Plant plausible mistakes in copies of the oracle; the pins must catch each.

Each mutant is a text substitution in oracle/hwr_oracle.c (a dropped term, a
wrong sign, index or operand, a swapped head, a changed rule), compiled on the
CPU into tests/_build/.  The test passes only if at least one pin check of
tests/pins.py fails on the mutant.  The oracle itself is never modified.
"""
import os

import pytest

import oracle
import pins

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "hwr_oracle.c")
BUILD = os.path.join(ROOT, "tests", "_build")

# (id, text in the oracle, replacement, how many occurrences to replace)
MUTANTS = [
    ("drop_b1", "double acc = m->b1[j];", "double acc = 0.0;", 1),
    ("drop_b1_f32", "float acc = m->b1[j];", "float acc = 0.0f;", 1),
    ("drop_b2", "double acc = m->b2[i];", "double acc = 0.0;", 1),
    ("drop_b3", "double acc = m->b3[o];", "double acc = 0.0;", 1),
    ("transpose_W1", "m->W1[(size_t)j * m->F + k]", "m->W1[(size_t)k * m->H1 + j]", 2),
    ("transpose_W2", "m->W2[(size_t)i * m->H1 + j]", "m->W2[(size_t)j * m->H2 + i]", 2),
    ("no_relu_h1", "h1[j] = acc > 0.0 ? acc : 0.0;", "h1[j] = acc;", 1),
    ("no_relu_h2_f32", "h2[i] = acc > 0.0f ? acc : 0.0f;", "h2[i] = acc;", 1),
    ("swap_heads", "*ttft = orc_softplus_f64(z[0]);\n    *tpot = orc_softplus_f64(z[1]);",
     "*ttft = orc_softplus_f64(z[1]);\n    *tpot = orc_softplus_f64(z[0]);", 1),
    ("softplus_drops_max", "return fmax(z, 0.0) + log1p(exp(-fabs(z)));",
     "return log1p(exp(-fabs(z)));", 1),
    ("sigmoid_sign", "return 1.0 / (1.0 + exp(-s));", "return 1.0 / (1.0 + exp(s));", 1),
    ("cost_sign", "double C = ttft + n * tpot;", "double C = ttft - n * tpot;", 1),
    ("cost_drops_ttft_f32", "float C = fmaf(n, tpot, ttft);", "float C = n * tpot;", 1),
    ("cost_uses_in_len", "double n = m->n_heads == 3 ? nout : (double)out_len;",
     "double n = m->n_heads == 3 ? nout : (double)in_len;", 1),
    ("utility_sign", "w->U[d] = wq * qual - (double)lam * C;",
     "w->U[d] = wq * qual + (double)lam * C;", 1),
    ("convex_weight", "double wq = convex ? 1.0 - (double)lam : 1.0;",
     "double wq = convex ? (double)lam : 1.0;", 1),
    ("quality_by_gpu", "double qual = w->qual[m->dep_model[d]];",
     "double qual = w->qual[m->dep_gpu[d]];", 1),
    ("quality_transposed", "(double)m->memb[(size_t)k * m->M + mi]",
     "(double)m->memb[(size_t)mi * m->E + k]", 1),
    ("running_reads_waiting", "if (k == P + 1) return (double)s->running[d];",
     "if (k == P + 1) return (double)s->waiting[d];", 1),
    ("gpu_onehot_offset", "return m->dep_gpu[d] == k - M ? 1.0 : 0.0;",
     "return m->dep_gpu[d] == k ? 1.0 : 0.0;", 1),
    ("in_out_swapped", "if (k == F - 2) return in_len;", "if (k == F - 2) return out_len;", 1),
    ("log1p_as_log", "if (code == 1) return log1p(v);", "if (code == 1) return log(v);", 1),
    ("standardise_multiplies", "double v = (t - (double)m->mu[k]) / (double)m->sd[k];",
     "double v = (t - (double)m->mu[k]) * (double)m->sd[k];", 1),
    ("slo_strict", "(C[d] <= slo);", "(C[d] < slo);", 1),
    ("slo_strict_f32", "((float)C[d] <= (float)slo)", "((float)C[d] < (float)slo)", 1),
    ("ties_to_highest", "(U[d] > U[best]);", "(U[d] >= U[best]);", 1),
    ("fallback_max_cost", "(C[d] < C[best]);", "(C[d] > C[best]);", 1),
    ("no_sequential_increment", "if (c >= 0) running_io[c] += 1;",
     "if (c >= 0) running_io[c] += 0;", 1),
    ("unfused_layer2_f32", "acc = fmaf(m->W2[(size_t)i * m->H1 + j], h1[j], acc);",
     "acc = acc + m->W2[(size_t)i * m->H1 + j] * h1[j];", 1),
    ("descending_layer1_f32",
     "for (int k = 0; k < m->F; ++k)\n            acc = fmaf(",
     "for (int k = m->F - 1; k >= 0; --k)\n            acc = fmaf(", 1),
    ("features_not_rounded_f32", "x[k] = mode == ORC_F32 ? (double)(float)v : v;",
     "x[k] = v;", 1),
    ("budget_drops_slack", "return (double)slack * ((double)a + (double)b * (double)p) +",
     "return ((double)a + (double)b * (double)p) +", 1),
    ("budget_order_f32", "float t = fmaf(b, p, a);\n    float s = slack * t;",
     "float t = b * p + a;\n    float s = slack * t;", 1),
    ("per_query_slo_first_only", "finish_query(m, &w, slo_q[q], mode,", "finish_query(m, &w, slo_q[0], mode,", 1),
    ("third_head_ignored", "double n = m->n_heads == 3 ? nout : (double)out_len;",
     "double n = (double)out_len;", 1),
    ("third_head_ignored_f32", "float n = m->n_heads == 3 ? nout : out_len;",
     "float n = out_len;", 1),
    ("third_head_reads_ttft", "*nout = m->n_heads == 3 ? orc_softplus_f64(z[2]) : 0.0;",
     "*nout = m->n_heads == 3 ? orc_softplus_f64(z[0]) : 0.0;", 1),
    ("per_query_seq_no_increment", "if (sequential && chosen[q] >= 0) running_io[chosen[q]] += 1;",
     "if (sequential && chosen[q] >= 0) running_io[chosen[q]] += 0;", 1),
]


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("mid,old,new,count", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(source, mid, old, new, count):
    assert source.count(old) == count, f"mutation site for {mid} not found"
    os.makedirs(BUILD, exist_ok=True)
    src = os.path.join(BUILD, f"mutant_{mid}.c")
    with open(src, "w") as f:
        f.write(source.replace(old, new))
    so = oracle.build(src=src, out=os.path.join(BUILD, f"libmutant_{mid}.so"))
    lib = oracle.load(path=so)
    caught = []
    for check in pins.ALL_CHECKS:
        try:
            check(lib)
        except AssertionError:
            caught.append(check.__name__)
            break
    assert caught, f"no pin detects mutant {mid}"
