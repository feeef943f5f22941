"""The oracle's second part against its pins, and the pins against mutated builds."""
import os
import subprocess
import tempfile

import pytest

import oracle as oracle_pkg
import oracle_pins_ext as pins


@pytest.fixture(scope="module")
def paper_oracle():
    return oracle_pkg.PaperOracle()


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_paper_oracle_pin(paper_oracle, check):
    check(paper_oracle)


# One plausible mistake per mutation, planted in a copy of lookme_oracle_ext.c.
MUTATIONS = {
    "silu_as_sigmoid": ("return x / (1.0 + exp(-x));", "return 1.0 / (1.0 + exp(-x));"),
    "ranker_centroid_half_on_v": ("acc += (double)w[de + k] * (double)ct[k];",
                                  "acc += (double)w[de + k] * (double)vt[k];"),
    "ranker_no_bf16_hidden": ("if (round_hidden) h[m] = to_bf16(h[m]);", ""),
    "ranker_drops_b2": ("double acc = (double)b2[p];", "double acc = 0.0;"),
    "ranker_drops_b1": ("double acc = (double)b1[m];", "double acc = 0.0;"),
    "level2_no_tanh": ("s[j] = cosv + tanh(rs[j].r);", "s[j] = cosv + rs[j].r;"),
    "level2_no_cos": ("s[j] = cosv + tanh(rs[j].r);", "s[j] = tanh(rs[j].r);"),
    "level2_dot_not_cos": ("const double cosv = (nv > 0.0 && nk > 0.0) ? dot / (nv * nk) : 0.0;",
                           "const double cosv = dot;"),
    "level2_ascending": ("if (x->r > y->r) return -1;\n    if (x->r < y->r) return 1;",
                         "if (x->r < y->r) return -1;\n    if (x->r > y->r) return 1;"),
    "level2_tie_higher_p": ("return (x->p < y->p) ? -1 : (x->p > y->p);", "return (x->p > y->p) ? -1 : (x->p < y->p);"),
    "gate_at_half_inclusive": ("gate[t] = acc > 0.0 ? 1 : 0;", "gate[t] = acc >= 0.0 ? 1 : 0;"),
    "text_ignores_gate": ("const int on = (!gate || gate[t]) && u >= 0 && u < V;", "const int on = u >= 0 && u < V;"),
    "text_no_range_check": ("const int on = (!gate || gate[t]) && u >= 0 && u < V;",
                            "const int on = (!gate || gate[t]) && u >= 0;"),
    "swiglu_roles_swapped": ("u[f] = silu(a) * b;", "u[f] = a * silu(b);"),
    "swiglu_no_round": ("if (round_mid) u[f] = to_bf16(u[f]);", ""),
    "propagate_transposed": ("(double)Wp[k * de + o]", "(double)Wp[o * de + k]"),
    "propagate_no_residual": ("double acc = (double)R[i * de + o];", "double acc = 0.0;"),
    "router_no_scale": ("s[m] = dot * inv;", "s[m] = dot;"),
    "router_transposed_projection": ("(double)Whe[k * de + o]", "(double)Whe[o * dh + k]"),
    "combine_first_weight_only": ("R[t * dv + d] += weight[t * T + j] * (double)row[d];",
                                  "R[t * dv + d] += weight[t * T] * (double)row[d];"),
}


@pytest.fixture(scope="module")
def mutant_dir():
    with tempfile.TemporaryDirectory() as d:
        yield d


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_ext_pins_reject_mutant(name, mutant_dir):
    old, new = MUTATIONS[name]
    with open(oracle_pkg._SRC_EXT) as f:
        src = f.read()
    assert src.count(old) >= 1, f"mutation {name}: pattern not found"
    path = os.path.join(mutant_dir, f"{name}.c")
    with open(path, "w") as f:
        f.write(src.replace(old, new, 1))
    so = os.path.join(mutant_dir, f"lib{name}.so")
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-fopenmp", path, "-o", so, "-lm"], check=True)
    bad = pins.failing_checks(oracle_pkg.PaperOracle(oracle_pkg.load_ext(so)))
    assert bad, f"mutation {name} survived every pin"
