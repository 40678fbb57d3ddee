"""Planted mistakes in the CPU oracle must be caught by its pins.

Each mutant is the oracle's source with one plausible mistake (a dropped term,
a wrong sign, index or axis, a reversed order, a strict instead of an
inclusive comparison, ...), loaded as a separate module on the CPU.  The test
passes when at least one pin of ``oracle_pins.ALL_CHECKS`` fails on it, which
shows that the pins constrain every step of the oracle.
"""
import importlib.util
import os
import sys
import types

import pytest

import oracle_pins as P

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "densitykv.py")

# (name, original text, mutated text)
MUTANTS = [
    ("w_exponent_sign", "np.power(prm.eps + np.asarray(d2, dtype=np.float64) / (s * s), -prm.p)",
     "np.power(prm.eps + np.asarray(d2, dtype=np.float64) / (s * s), prm.p)"),
    ("w_sigma_not_squared", "np.power(prm.eps + np.asarray(d2, dtype=np.float64) / (s * s), -prm.p)",
     "np.power(prm.eps + np.asarray(d2, dtype=np.float64) / s, -prm.p)"),
    ("w_eps_dropped", "np.power(prm.eps + np.asarray(d2, dtype=np.float64) / (s * s), -prm.p)",
     "np.power(1.0 + np.asarray(d2, dtype=np.float64) / (s * s), -prm.p)"),
    ("sigma_default", "math.sqrt(d / 2.0) if self.sigma is None", "math.sqrt(d) if self.sigma is None"),
    ("dist_cross_factor", "na[:, None] + nb[None, :] - 2.0 * (A @ B.T)", "na[:, None] + nb[None, :] - (A @ B.T)"),
    ("dist_wrong_norm", "na[:, None] + nb[None, :] - 2.0 * (A @ B.T)", "na[:, None] + na[:, None] - 2.0 * (A @ B.T)"),
    ("density_includes_self", "    W[np.arange(n), np.arange(n)] = 0.0", "    pass"),
    ("score_times_b", "(Wxb / hb.base.astype(np.float64)[None, :])", "(Wxb * hb.base.astype(np.float64)[None, :])"),
    ("score_no_mean", ".sum(axis=1) / m\n", ".sum(axis=1)\n"),
    ("sort_descending", 'pi = np.argsort(s, kind="stable")', 'pi = np.argsort(-s, kind="stable")'),
    ("sort_ties_reversed", 'pi = np.argsort(s, kind="stable")',
     'pi = (len(s) - 1 - np.argsort(s[::-1], kind="stable"))'),
    ("prefix_reversed", "np.cumsum(Wmat, axis=1)", "np.cumsum(Wmat[:, ::-1], axis=1)"),
    ("prefix_drops_rho", "out[:, 1:] = hb.rho.astype(np.float64)[:, None] + np.cumsum(Wmat, axis=1)",
     "out[:, 1:] = np.cumsum(Wmat, axis=1)"),
    ("violation_strict", "viol = g >= prm.tau", "viol = g > prm.tau"),
    ("evict_budget_off_by_one", "e = np.maximum(0, m + r_all - hb.M)", "e = np.maximum(0, m + r_all - hb.M + 1)"),
    ("rstar_min", "r_star = int(np.nonzero(allf)[0].max())", "r_star = int(np.nonzero(allf)[0].min())"),
    ("rstar_any_head", "allf = np.logical_and.reduce(", "allf = np.logical_or.reduce("),
    ("mandatory_at_zero", "mand = (g_r >= prm.tau) if r > 0", "mand = (g[:, 0] >= prm.tau) if r > 0"),
    ("fill_sparsest", "order = np.lexsort((hb.src[rest], hb.step[rest], -rho_t[rest]))",
     "order = np.lexsort((hb.src[rest], hb.step[rest], rho_t[rest]))"),
    ("fill_ties_newest", "order = np.lexsort((hb.src[rest], hb.step[rest], -rho_t[rest]))",
     "order = np.lexsort((-hb.src[rest], -hb.step[rest], -rho_t[rest]))"),
    ("survivor_no_subtract", "rho_surv = rho_t[keep] - sub", "rho_surv = rho_t[keep]"),
    ("survivor_no_admitted", "rho_surv = rho_t[keep] - sub", "rho_surv = hb.rho.astype(np.float64)[keep] - sub"),
    ("new_includes_self", "            W_new[np.arange(r), n_surv + np.arange(r)] = 0.0                  # exclude self by index",
     "            pass"),
    ("new_excludes_coadmitted", "W_new = soft_riesz(sq_dist(K_new[n_surv:], K_new), prm, hb.d)",
     "W_new = soft_riesz(sq_dist(K_new[n_surv:], np.concatenate([K_new[:n_surv], K_new[n_surv:] + 1e9])), prm, hb.d)"),
    ("baseline_floor_min", "np.maximum(rho_new, prm.delta)]", "np.minimum(rho_new, prm.delta)]"),
    ("baseline_refreshed", "hb.base = np.concatenate([hb.base[keep],", "hb.base = np.concatenate([np.maximum(rho_surv, prm.delta),"),
    ("init_last_candidates", "hb.K = np.asarray(Kc[:r], dtype=np.float64).copy()",
     "hb.K = np.asarray(Kc[N - r:], dtype=np.float64).copy()"),
    ("values_unpaired", "V_new = np.concatenate([hb.V[keep], Vc[h][adm]], axis=0)",
     "V_new = np.concatenate([hb.V[keep], Vc[h][np.sort(adm)]], axis=0)"),
    ("attn_no_scale", "S = (Q @ Kall.T) / math.sqrt(Q.shape[1])", "S = (Q @ Kall.T)"),
    ("attn_wrong_axis", "P /= P.sum(axis=1, keepdims=True)", "P /= P.sum(axis=0, keepdims=True)"),
    ("attn_drops_window", "Kall = np.concatenate([hb.K, np.asarray(Kw, dtype=np.float64)], axis=0)",
     "Kall = np.concatenate([hb.K, 0.0 * np.asarray(Kw, dtype=np.float64)], axis=0)"),
    ("storage_meta", "meta_bytes: int = 4 + 4 + 8 + 4", "meta_bytes: int = 4 + 4 + 4 + 4"),
    ("densest_ascending", "order = np.lexsort((hb.src, hb.step, -rho_t))",
     "order = np.lexsort((hb.src, hb.step, rho_t))"),
    ("source_fill_newest_first", "order = np.lexsort((hb.src[rest], hb.step[rest]))\n",
     "order = np.lexsort((-hb.src[rest], -hb.step[rest]))\n"),
    ("refresh_ignored", "if prm.refresh_baselines:\n", "if False:\n"),
    ("source_order_ignored", 'if prm.order == "score" else np.arange(N)', 'if True else np.arange(N)'),
    ("densest_keeps_mandatory_first", 'if prm.evict == "densest":', 'if prm.evict == "never":'),
    ("sequential_source_order", "        c = pi[:, j]\n", "        c = np.arange(H) * 0 + j\n"),
    ("sequential_src_dropped", "adm_src = adm if src_index is None else np.asarray(src_index[h])[adm]",
     "adm_src = adm"),
    ("block_order_descending", '        out[h] = np.argsort(s, kind="stable")', '        out[h] = np.argsort(-s, kind="stable")'),
    ("rope_x_sign", "out[:, :, xi] = x * c + y * s", "out[:, :, xi] = x * c - y * s"),
    ("rope_y_sign", "out[:, :, yi] = y * c - x * s", "out[:, :, yi] = y * c + x * s"),
    ("rope_half_as_interleaved", "        xi, yi = np.arange(d // 2), np.arange(d // 2, d)",
     "        xi, yi = np.arange(0, d, 2), np.arange(1, d, 2)"),
    ("rope_first_token_time", "a = t[:, None] * th[None, :]", "a = t[:1, None] * th[None, :]"),
    ("bf16_ties_up", "out = np.ldexp(np.rint(m * 256.0), e - 8)", "out = np.ldexp(np.floor(m * 256.0 + 0.5), e - 8)"),
    ("bf16_through_fp32", "m, e = np.frexp(x)", "m, e = np.frexp(x.astype(np.float32).astype(np.float64))"),
    ("kv_keys_only", "    return np.concatenate([np.asarray(K, dtype=np.float64), np.asarray(V, dtype=np.float64)], axis=-1)",
     "    return np.concatenate([np.asarray(K, dtype=np.float64), 0.0 * np.asarray(V, dtype=np.float64)], axis=-1)"),
    ("kv_value_twice", "    return np.concatenate([np.asarray(K, dtype=np.float64), np.asarray(V, dtype=np.float64)], axis=-1)",
     "    return np.concatenate([np.asarray(V, dtype=np.float64), np.asarray(V, dtype=np.float64)], axis=-1)"),
]


def _load_mutant(name, old, new):
    src = open(SRC).read()
    assert src.count(old) >= 1, f"mutation anchor not found for {name}"
    mod = types.ModuleType(f"oracle_mutant_{name}")
    mod.__file__ = SRC
    sys.modules[mod.__name__] = mod
    exec(compile(src.replace(old, new, 1), f"<mutant {name}>", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(name, old, new):
    mod = _load_mutant(name, old, new)
    failed = []
    for check in P.ALL_CHECKS:
        try:
            check(mod)
        except Exception as exc:  # an assertion or a crash both reveal the mistake
            failed.append((check.__name__, type(exc).__name__))
    assert failed, f"mutant {name} passed every pin"
