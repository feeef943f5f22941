"""The CPU oracle against its pins, and the pins against mutated oracles."""
import os
import subprocess
import tempfile

import pytest

import oracle as oracle_pkg
import oracle_pins as pins


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_oracle_pin(oracle, check):
    check(oracle)


# Each mutation plants one plausible mistake in a copy of the oracle's C source.
# The pin suite must reject every one of them.
MUTATIONS = {
    "route_drops_bias": ("score = cosv + (bias ? (double)bias[s] : 0.0)", "score = cosv + 0.0"),
    "route_dot_not_cosine": ("dot / (nt * cnorm[s])", "dot"),
    "route_no_query_norm": ("dot / (nt * cnorm[s])", "dot / cnorm[s]"),
    "route_tie_takes_last": ("if (score > best) {", "if (score >= best) {"),
    "centroid_wrong_divisor": ("acc / (double)P", "acc / (double)(P + 1)"),
    "level2_no_temperature": ("zs[p].z = dot * inv_sqrt_dk;", "zs[p].z = dot;"),
    "level2_ascending": ("if (x->z > y->z) return -1;\n    if (x->z < y->z) return 1;",
                         "if (x->z < y->z) return -1;\n    if (x->z > y->z) return 1;"),
    "level2_tie_higher_p": ("return (x->p < y->p) ? -1 : (x->p > y->p);",
                            "return (x->p > y->p) ? -1 : (x->p < y->p);"),
    "level2_wrong_scene": ("const float* Kj = key_blocks + block_of_scene[scene[t]] * P * dk;\n            for (int64_t p",
                           "const float* Kj = key_blocks + block_of_scene[0] * P * dk;\n            for (int64_t p"),
    "level2_softmax_over_all": ("for (int32_t j = 0; j < top_k; ++j)\n                denom += exp(zs[j].z - zmax);",
                                "for (int32_t j = 0; j < P; ++j)\n                denom += exp(zs[j].z - zmax);"),
    "level2_transposed_key": ("(double)Kj[p * dk + d];\n                zs[p].z", "(double)Kj[d * P + p];\n                zs[p].z"),
    "select_ceil": ("(int64_t)floor((double)len * keep_ratio)", "(int64_t)ceil((double)len * keep_ratio)"),
    "select_tie_higher_t": ("return (x->t < y->t) ? -1 : (x->t > y->t);", "return (x->t > y->t) ? -1 : (x->t < y->t);"),
    "select_smallest": ("if (x->pi > y->pi) return -1;", "if (x->pi < y->pi) return -1;"),
    "inject_first_weight_only": ("R[d] += weight[t * top_k + j] * (double)row[d];", "R[d] += weight[t * top_k] * (double)row[d];"),
    "inject_prim_as_scene": ("const float* row = Vj + (int64_t)prim[t * top_k + j] * dv;",
                             "const float* row = value_blocks + (int64_t)prim[t * top_k + j] * dv;"),
    "round_truncates": ("r = ldexp(nearbyint(ldexp(m, 8)), e - 8);", "r = ldexp(floor(ldexp(m, 8)), e - 8);"),
}


@pytest.fixture(scope="module")
def mutant_dir():
    with tempfile.TemporaryDirectory() as d:
        yield d


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_reject_mutant(name, mutant_dir):
    old, new = MUTATIONS[name]
    with open(oracle_pkg._SRC) as f:
        src = f.read()
    assert src.count(old) >= 1, f"mutation {name}: pattern not found in the oracle source"
    mutated = src.replace(old, new, 1)
    path = os.path.join(mutant_dir, f"{name}.c")
    with open(path, "w") as f:
        f.write(mutated)
    so = os.path.join(mutant_dir, f"lib{name}.so")
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-fopenmp", path, "-o", so, "-lm"], check=True)
    bad = pins.failing_checks(oracle_pkg.Oracle(oracle_pkg.load(so)))
    assert bad, f"mutation {name} survived every pin"
