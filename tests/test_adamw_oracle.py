"""The fp64 AdamW oracle against its pins, and planted mistakes in a copy of
it caught by them (CPU only)."""
import inspect
import sys
import types

import pytest

import oracle.adamw_ref as ref
from tests import adamw_pins


@pytest.mark.parametrize("check", adamw_pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_adamw_pin(check):
    check(ref)


MUTATIONS = {
    "no_bias_correction_v": ("v_hat = state.v / (1.0 - hp.beta2 ** t)", "v_hat = state.v"),
    "no_bias_correction_m": ("m_hat = state.m / (1.0 - hp.beta1 ** t)", "m_hat = state.m"),
    "eps_inside_sqrt": ("(np.sqrt(v_hat) + hp.eps)", "np.sqrt(v_hat + hp.eps)"),
    "betas_swapped": ("state.m = hp.beta1 * state.m + (1.0 - hp.beta1) * g",
                      "state.m = hp.beta2 * state.m + (1.0 - hp.beta2) * g"),
    "coupled_decay": ("g = np.asarray(g, dtype=np.float64)",
                      "g = np.asarray(g, dtype=np.float64) + weight_decay * np.asarray(w)"),
    "decay_after_step": ("w_new = (1.0 - hp.lr * weight_decay) * w - update",
                         "w_new = (1.0 - hp.lr * weight_decay) * (w - update)"),
    "t_not_incremented": ("state.t += 1", "state.t += 0"),
    "v_not_squared": ("(1.0 - hp.beta2) * g * g", "(1.0 - hp.beta2) * np.abs(g)"),
    "decay_sign": ("(1.0 - hp.lr * weight_decay) * w", "(1.0 + hp.lr * weight_decay) * w"),
}


def _mutant(old, new):
    src = inspect.getsource(ref)
    assert src.count(old) == 1, f"mutation anchor not found once: {old!r}"
    name = "adamw_mutant_%d" % abs(hash((old, new)))
    mod = types.ModuleType(name)
    sys.modules[name] = mod
    exec(compile(src.replace(old, new), name, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name):
    mod = _mutant(*MUTATIONS[name])
    caught = []
    for check in adamw_pins.ALL_CHECKS:
        try:
            check(mod)
        except Exception as e:
            caught.append((check.__name__, type(e).__name__))
    assert caught, f"no pin caught mutation {name}"
