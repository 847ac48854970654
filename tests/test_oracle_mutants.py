"""Pin strength: each plausible mistake planted in a copy of the oracle
(a swapped operand, a dropped term, a wrong index or sign, a non-strict
comparison) must make at least one oracle pin fail.  The mutants are built
on the CPU from osd_oracle.c by one textual replacement each and run the pin
suites in a subprocess; the real oracle is untouched."""
import os
import subprocess
import sys

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
SRC = os.path.join(ROOT, "oracle", "osd_oracle.c")

# (name, original text, mutated text, occurrence count to replace)
MUTANTS = [
    ("residual_operands_swapped", "double d = exp(lp[j]) - exp(lq[j]);",
     "double d = exp(lq[j]) - exp(lp[j]);", 1),
    ("accept_not_strict", "if (u[a] < r) ++a;", "if (u[a] <= r) ++a;", 1),
    ("sample_uses_wrong_uniform", "double tau = u[k] * W;", "double tau = u[a] * W;", 1),
    ("cdf_not_strict", "if (C > tau) { sample = j; break; }",
     "if (C >= tau) { sample = j; break; }", 1),
    ("draft_temperature_dropped", "log_softmax(draft + (b * k + a) * V, V, T, lq);",
     "log_softmax(draft + (b * k + a) * V, V, 1.0, lq);", 2),
    ("bonus_from_last_draft_position", "log_softmax(target + (b * (k + 1) + a) * V, V, T, lp);\n            if (a < k)",
     "log_softmax(target + (b * (k + 1) + (a < k ? a : k - 1)) * V, V, T, lp);\n            if (a < k)", 1),
    ("argmax_last_on_ties", "if (x[j] > x[best]) best = j;", "if (x[j] >= x[best]) best = j;", 1),
    ("mask_off_by_one", "if (a < k) mask[b * k + a] = 1;", "if (a > 0) mask[b * k + a - 1] = 1;", 1),
    ("lse_without_max", "double lse = m + log(sum);", "double lse = log(sum);", 1),
    ("fkl_grad_sign", "g[j] = exp(lq[j]) - exp(lp[j]);", "g[j] = exp(lp[j]) - exp(lq[j]);", 1),
    ("rkl_grad_drops_loss", "q * ((lq[j] - lp[j]) - l)", "q * (lq[j] - lp[j])", 1),
    ("rkl_is_fkl", "if (q > 0.0) l += q * (lq[j] - lp[j]);",
     "if (q > 0.0) l += exp(lp[j]) * (lp[j] - lq[j]);", 1),
    ("jsd_mixture_weights_swapped", "double m = beta * p + (1.0 - beta) * q;",
     "double m = (1.0 - beta) * p + beta * q;", 2),
    ("jsd_grad_uses_klp", "(log(q / m) - klq)", "(log(q / m) - klp)", 1),
    ("tvd_sign_flipped", "double s = (q > p) ? 0.5 : (q < p ? -0.5 : 0.0);",
     "double s = (q < p) ? 0.5 : (q > p ? -0.5 : 0.0);", 2),
    ("tvd_half_dropped", "l += 0.5 * fabs(p - q);", "l += fabs(p - q);", 1),
    ("temperature_factor_dropped", "for (long j = 0; j < V; ++j) g[j] /= tau;", "", 1),
    ("ce_label_from_draft", "long ystar = argmax_first(target + n * V, V);",
     "long ystar = argmax_first(draft + n * V, V);", 1),
    ("distill_temperature_ignored", "log_softmax(target + n * V, V, tau, lp);",
     "log_softmax(target + n * V, V, 1.0, lp);", 1),
    ("mixture_weights_swapped", "w[j] = beta * exp(lp[j]) + (1.0 - beta) * exp(lq[j]);",
     "w[j] = (1.0 - beta) * exp(lp[j]) + beta * exp(lq[j]);", 1),
    ("mixture_temperature_ignored", "log_softmax(draft + n * d_stride, V, tau, lq);",
     "log_softmax(draft + n * d_stride, V, 1.0, lq);", 1),
    ("mixture_cdf_not_strict", "if (C > target_mass) { pick = j; break; }",
     "if (C >= target_mass) { pick = j; break; }", 1),
    ("mixture_target_only", "w[j] = beta * exp(lp[j]) + (1.0 - beta) * exp(lq[j]);",
     "w[j] = exp(lp[j]);", 1),
    ("tree_residual_not_updated", "const double d = r[j] - q[j];", "const double d = r[j];", 1),
    ("tree_siblings_reversed",
     "for (long c = node + 1; c < n_nodes && next < 0; ++c) {\n                    if (parent[c] != node) continue;",
     "for (long c = n_nodes - 1; c > node && next < 0; --c) {\n                    if (parent[c] != node) continue;", 1),
    ("tree_extra_uses_node_uniform", "const double mass = u[0] * W;", "const double mass = u[node] * W;", 1),
    ("tree_ratio_inverted", "if (qy > 0.0) ratio = ry / qy;", "if (ry > 0.0) ratio = qy / ry;", 1),
]


@pytest.mark.parametrize("name,old,new,count", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, name, old, new, count):
    src = open(SRC).read()
    assert src.count(old) == count, f"mutation site for {name} not found"
    mutant = tmp_path / f"{name}.c"
    mutant.write_text(src.replace(old, new))
    lib = oracle.compile_source(str(mutant), str(tmp_path / f"lib{name}.so"))
    env = dict(os.environ, OSD_ORACLE_LIB=lib)
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(HERE, "test_oracle_distill.py"),
                        os.path.join(HERE, "test_oracle_verify.py"),
                        os.path.join(HERE, "test_oracle_mixed.py"),
                        os.path.join(HERE, "test_oracle_tree.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 1, f"mutant {name} survived every pin:\n{r.stdout[-2000:]}"
