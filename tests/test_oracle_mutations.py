"""Plant plausible mistakes in a copy of the oracle (on the CPU) and show that
the pins catch each one: a dropped term, a wrong sign, a swapped operand or
index, a wrong constant."""
import inspect
import sys
import types

import pytest

import oracle.malt_ref as ref
from tests import oracle_pins

MUTATIONS = {
    "exponent_quarter": ("PRECOND_EXPONENT = -1.0 / 8.0", "PRECOND_EXPONENT = -1.0 / 4.0"),
    "momentum_uses_mu2": ("state.M = ema(state.M, G, hp.mu1)", "state.M = ema(state.M, G, hp.mu2)"),
    "row_col_swapped": ("return np.sum(G * G, axis=1), np.sum(G * G, axis=0)",
                        "return np.sum(G * G, axis=0), np.sum(G * G, axis=1)"),
    "backmap_LR_swapped": ("D = two_sided(Ld, O, Rd)", "D = two_sided(Rd, O, Ld)"),
    "backmap_dropped": ("D = two_sided(Ld, O, Rd)", "D = O"),
    "ns_sign_flip": ("B = b * A + c * (A @ A)", "B = b * A - c * (A @ A)"),
    "ns_no_normalise": ("X = X / (np.linalg.norm(X) + ns_eps)", "X = X"),
    "ns_no_transpose_back": ("return X.T if transposed else X", "return X"),
    "graft_drops_normO": ("scale = hp.lr * norm_O / (norm_D + hp.eps)",
                          "scale = hp.lr / (norm_D + hp.eps)"),
    "malter_bias_mu1_fixed": ("(1.0 - hp.mu1 ** t + hp.eps)", "(1.0 - hp.mu1 + hp.eps)"),
    "malter_nu_uses_M": ("lgr_sq = float(np.sum(two_sided(Ld, G, Rd) ** 2))",
                         "lgr_sq = float(np.sum(two_sided(Ld, state.M, Rd) ** 2))"),
    "malter_sqrt_dropped": ("math.sqrt(1.0 - hp.mu2 ** t)", "(1.0 - hp.mu2 ** t)"),
    "bf16_one_bit_short": ("np.maximum(e - 8, -133)", "np.maximum(e - 9, -133)"),
    "t_not_incremented": ("state.t += 1 ", "state.t += 0 "),
    "lr_twice_in_malter": ("scale *= alpha", "scale *= alpha * hp.lr"),
    "ns_gram_transposed": ("A = X @ X.T", "A = X.T @ X"),
    "ns_product_order": ("X = a * X + B @ X", "X = a * X + X @ B"),
    "ns_linear_coeff_dropped": ("X = a * X + B @ X", "X = X + B @ X"),
    "eps_outside_root": ("np.power(np.asarray(v, dtype=np.float64) + eps, PRECOND_EXPONENT)",
                         "np.power(np.asarray(v, dtype=np.float64), PRECOND_EXPONENT) + eps"),
    "ema_weights_swapped": ("return mu * prev + (1.0 - mu) * new",
                            "return (1.0 - mu) * prev + mu * new"),
    "two_sided_diagonals_swapped": ("return Ld[:, None] * X * Rd[None, :]",
                                    "return Ld[None, :] * X * Rd[:, None]"),
    "alpha_uses_M_not_Mt": ("* norm_Mt / (math.sqrt(state.nu) + hp.eps))",
                            "* float(np.linalg.norm(state.M)) / (math.sqrt(state.nu) + hp.eps))"),
    "weight_decay_sign": ("(1.0 - hp.lr * hp.weight_decay) * W if",
                          "(1.0 + hp.lr * hp.weight_decay) * W if"),
    "weight_decay_after_update": ("W_new = W_decayed - delta",
                                  "W_new = (1.0 - hp.lr * hp.weight_decay) * (W - delta)"),
    "ns_scalar_map_wrong_power": ("x = a * x + b * x ** 3 + c * x ** 5",
                                  "x = a * x + b * x ** 3 + c * x ** 4"),
    "ns_scalar_map_coeffs_swapped": ("x = a * x + b * x ** 3 + c * x ** 5",
                                     "x = a * x + c * x ** 3 + b * x ** 5"),
    "graft_uses_normD_twice": ("scale = hp.lr * norm_O / (norm_D + hp.eps)",
                               "scale = hp.lr * norm_D / (norm_D + hp.eps)"),
}


def _mutant(old, new):
    src = inspect.getsource(ref)
    assert src.count(old) >= 1, f"mutation anchor not found: {old!r}"
    name = "oracle_mutant_%d" % abs(hash((old, new)))
    mod = types.ModuleType(name)
    sys.modules[name] = mod          # dataclasses resolve annotations through it
    exec(compile(src.replace(old, new), name, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name):
    mod = _mutant(*MUTATIONS[name])
    caught = []
    for check in oracle_pins.ALL_CHECKS:
        try:
            check(mod)
        except Exception as e:  # AssertionError or a shape error
            caught.append((check.__name__, type(e).__name__))
    assert caught, f"no pin caught mutation {name}"
