"""Planted mistakes in the oracle's protocol layer are caught by the pins (no GPU).

``test_oracle_mutants.py`` plants slips in the C source of the elementwise
rules.  This file does the same for the Python layer of ``oracle/__init__.py``
that turns them into the server of Sec. 2.1-2.3: the FIFO of pushes, the
staleness tau = T - j a push finds, the per-client push and fetch counters
that key the draws, the per-message gradient cache and the per-tensor
decisions.  Each mutant is the module's source with one plausible slip,
loaded as a separate module; the pins then run against it (``pins.oracle``
is pointed at the mutant for the test) and at least one must fail.
"""

import types

import pytest

import oracle
import pins

PY_MUTANTS = {
    # protocol order and staleness (Sec. 2.1)
    "fifo_last_first": ("kind, client, j, payload = self.fifo.pop(0)",
                        "kind, client, j, payload = self.fifo.pop()"),
    "tau_off_by_one": ("tau = self.T - j", "tau = self.T - j + 1"),
    "future_timestamp_accepted": ("if not 0 <= j <= self.T:", "if not 0 <= j <= self.T + 1:"),
    # per-message rule (Sec. 2.3): counter, stream, cache, statistic
    "message_push_counter_stuck": (
        "                n = self.push_count[client]\n"
        "                self.push_count[client] += 1\n"
        "                u = draw_message(self.seed, 0, client, n)",
        "                n = self.push_count[client]\n"
        "                u = draw_message(self.seed, 0, client, n)"),
    "message_push_fetch_stream": ("u = draw_message(self.seed, 0, client, n)",
                                  "u = draw_message(self.seed, 1, client, n)"),
    "message_drop_applies_new": ("                if sent:\n"
                                 "                    self.cache[client] = payload.copy()",
                                 "                self.cache[client] = payload.copy()"),
    "message_cache_one_slot": ("self.cache[client] = payload.copy()",
                               "self.cache[0] = payload.copy()"),
    "message_mean_of_theta": ("                vbar = mean_v(self.v, self.real)\n"
                              "                sent = decide(",
                              "                vbar = mean_v(self.theta, self.real)\n"
                              "                sent = decide("),
    "fetch_message_counter_stuck": (
        "        n = self.fetch_count[client]\n"
        "        self.fetch_count[client] += 1\n"
        "        u = draw_message(self.seed, 1, client, n)",
        "        n = self.fetch_count[client]\n"
        "        u = draw_message(self.seed, 1, client, n)"),
    "fetch_message_always_copies": ("        if ok:\n            theta_client[:] = self.theta",
                                    "        if True:\n            theta_client[:] = self.theta"),
    # per-parameter rule: the counters that key the draws
    "select_counter_stuck": ("        self.push_count[client] += 1\n        return out",
                             "        return out"),
    "fetch_compact_push_counter": ("self.seed, client, self.fetch_count[client],",
                                   "self.seed, client, self.push_count[client],"),
    # per-tensor rule under a budget
    "budget_push_counter_stuck": (
        "                n = self.push_count[client]\n"
        "                self.push_count[client] += 1\n"
        "                sent, cb, m = self._budget_decide(0, client, n, budget)",
        "                n = self.push_count[client]\n"
        "                sent, cb, m = self._budget_decide(0, client, n, budget)"),
    "budget_fetch_push_stream": ("sent, c, m = self._budget_decide(1, client, n, budget)",
                                 "sent, c, m = self._budget_decide(0, client, n, budget)"),
    "budget_fetch_copies_all": ("for t in np.flatnonzero(sent):",
                                "for t in range(sent.size):"),
    # the wrappers around the C rules: argument order, streams, counts
    "select_swaps_grad_and_v": ("ora_select(P, _ptr(g), _ptr(v), c,", "ora_select(P, _ptr(v), _ptr(g), c,"),
    "fetch_select_swaps_theta_and_v": ("ora_fetch_select(P, _ptr(th), _ptr(v), c,",
                                       "ora_fetch_select(P, _ptr(v), _ptr(th), c,"),
    "fetch_apply_applies_nothing": ("ora_fetch_apply(_ptr(theta_client), i.shape[0], _ptr(i), _ptr(x))",
                                    "ora_fetch_apply(_ptr(theta_client), 0, _ptr(i), _ptr(x))"),
    "draw_message_one_stream": ("ora_draw_message(seed, stream, client, n)",
                                "ora_draw_message(seed, 0, client, n)"),
    "tensor_select_one_stream": ("                                                stream, client, n, _ptr(sent))",
                                 "                                                0, client, n, _ptr(sent))"),
    "budget_c_half_budget": ("_ptr(vb), eps_b,\n                                                     int(budget)))",
                             "_ptr(vb), eps_b,\n                                                     int(budget) // 2))"),
    "sim_grad_one_client": ("seed, client,\n                                       n, _ptr(g))",
                            "seed, 0,\n                                       n, _ptr(g))"),
}


def _load_mutant(name, old, new):
    src = open(oracle.__file__).read()
    assert src.count(old) == 1, f"mutant {name}: pattern not (uniquely) in the oracle module"
    mod = types.ModuleType(f"oracle_protocol_mutant_{name}")
    mod.__file__ = oracle.__file__
    exec(compile(src.replace(old, new, 1), oracle.__file__, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(PY_MUTANTS))
def test_protocol_mutant_is_caught(monkeypatch, name):
    old, new = PY_MUTANTS[name]
    mutant = _load_mutant(name, old, new)
    monkeypatch.setattr(pins, "oracle", mutant)
    libs = pins.real_libs()
    caught = None
    for check in pins.ALL_CHECKS:   # the first pin that fails catches the mutant
        try:
            check(libs)
        except Exception as e:      # any failure of a pin counts as a catch
            caught = f"{check.__name__}: {type(e).__name__}"
            break
    assert caught is not None, f"protocol mutant {name} passed every pin"


def test_unmutated_module_passes_every_pin(monkeypatch):
    """The harness itself: the module loaded the same way, unchanged, passes."""
    monkeypatch.setattr(pins, "oracle", _load_mutant("none", "ASGD, SASGD, FASGD, FASGD_STD = 0, 1, 2, 3",
                                                     "ASGD, SASGD, FASGD, FASGD_STD = 0, 1, 2, 3"))
    libs = pins.real_libs()
    for check in pins.ALL_CHECKS:
        check(libs)


# The closed-loop simulation's oracle (oracle/sim.py): dispatcher batches,
# clients' stale copies and the timestamps they push with, the refreshes.
SIM_MUTANTS = {
    "sim_copy_timestamp_kept": ("                self.clients[c][:] = self.srv.theta.astype(np.float32)\n"
                                "                self.client_T[c] = T\n",
                                "                self.clients[c][:] = self.srv.theta.astype(np.float32)\n"),
    "sim_pushes_timestamp_zero": ("self.srv.push(c, self.client_T[c], g)", "self.srv.push(c, 0, g)"),
    "sim_grad_count_stuck": ("            self.grad_count[c] += 1\n", ""),
    "sim_grad_one_stream": ("g = sim_grad(self.clients[c], self.h, self.star, self.sigma, self.seed, c,",
                            "g = sim_grad(self.clients[c], self.h, self.star, self.sigma, self.seed, 0,"),
    "sim_param_fetch_dropped": ("                fetch_apply(self.clients[c], idx, val, lib=self.lib)\n", ""),
    "sim_message_timestamp_always": ("                if self.srv.fetch_message(c, self.clients[c]):\n"
                                     "                    self.client_T[c] = T",
                                     "                self.srv.fetch_message(c, self.clients[c])\n"
                                     "                self.client_T[c] = T"),
    "sim_budget_fetch_wrong_copy": ("self.srv.fetch_budget(c, self.clients[c], self.fetch_budget)",
                                    "self.srv.fetch_budget(c, self.clients[0], self.fetch_budget)"),
}


def _load_sim_mutant(name, old, new):
    import oracle.sim as osim
    src = open(osim.__file__).read()
    assert src.count(old) == 1, f"mutant {name}: pattern not (uniquely) in oracle/sim.py"
    mod = types.ModuleType(f"oracle_sim_mutant_{name}")
    mod.__file__ = osim.__file__
    mod.__package__ = "oracle"
    exec(compile(src.replace(old, new, 1), osim.__file__, "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(SIM_MUTANTS))
def test_sim_mutant_is_caught(monkeypatch, name):
    import sys
    old, new = SIM_MUTANTS[name]
    mutant = _load_sim_mutant(name, old, new)
    monkeypatch.setitem(sys.modules, "oracle.sim", mutant)
    monkeypatch.setattr(oracle, "sim", mutant, raising=False)
    libs = pins.real_libs()
    caught = None
    for check in pins.ALL_CHECKS:
        try:
            check(libs)
        except Exception as e:
            caught = f"{check.__name__}: {type(e).__name__}"
            break
    assert caught is not None, f"simulation mutant {name} passed every pin"
