"""Closed-loop simulation of asynchronous training on the CUDA path.

A stand-in for the paper's FRED simulator (Sec. 3): lambda clients hold their
own copies of the parameters, a dispatcher decides which clients push next
(``streams.dispatch_schedule``), each pushing client computes a stochastic
gradient of a synthetic quadratic at its (stale) copy, the server applies the
pushes in arrival order (ASGD / SASGD / FASGD / divide-by-std), and each
pushing client then refreshes its copy -- fully (``fetch="full"``), per
parameter through B-FASGD's fetch compaction (``"param"``), through one
per-message B-FASGD decision (``"message"``), or per tensor under a bandwidth
budget (``"budget"``: ``fetch_budget`` expected parameters per fetch over the
partition ``tensor_sizes``).  With ``push_budget`` the pushes, too, go per
tensor under that budget.  Everything on the device runs in the library's
kernels, through the C ABI.

Run as a script to compare the update rules over a learning-rate sweep:
``python -m paper_1601_04033_gb300.sim --compare``.
"""

from __future__ import annotations

import argparse
import json
import time

import numpy as np

from . import fasgd, streams


class Simulation:
    def __init__(self, P: int, lam: int, alpha: float, variant: int, *, K: int = 1,
                 gamma: float = 0.95, beta: float = 0.95, eps: float = 1e-4, seed: int = 0,
                 fetch: str = "full", c_fetch: float = 0.0, objective=None, theta0=None,
                 exact: bool = False, device: str = "cuda", eps_b: float = 1e-8,
                 tensor_sizes=None, fetch_budget: int | None = None,
                 push_budget: int | None = None):
        import torch
        if fetch not in ("full", "param", "message", "budget"):
            raise ValueError("fetch must be full, param, message or budget")
        if (fetch == "budget" and fetch_budget is None) or \
                ((fetch == "budget" or push_budget is not None) and tensor_sizes is None):
            raise ValueError("per-tensor budgets need tensor_sizes (and fetch_budget)")
        self.fetch_budget, self.push_budget = fetch_budget, push_budget
        self.torch = torch
        self.P, self.lam, self.K, self.seed, self.fetch = P, lam, K, seed, fetch
        self.stream = torch.cuda.current_stream()
        self.srv = fasgd.Server(P, lam, alpha, variant, gamma=gamma, beta=beta, eps=eps,
                                eps_b=eps_b, seed=seed, stream=self.stream)
        if tensor_sizes is not None:
            self.srv.set_tensors(tensor_sizes)
        self.srv.set_fetch_threshold(c_fetch)
        self.srv.set_exact(exact)
        h, star, sigma = objective if objective is not None else streams.quadratic_objective(seed, P)
        th0 = theta0 if theta0 is not None else np.zeros(P, np.float32)
        self._obj_buf, (self.h, self.star, self.sigma) = fasgd.aligned_vectors(
            np.stack([h, star, sigma]), device)
        self.srv.set_params(torch.from_numpy(np.ascontiguousarray(th0, np.float32)).to(device))
        self._cl_buf, self.clients = fasgd.aligned_vectors(np.tile(th0, (lam, 1)), device)
        self._g_buf, self.grads = fasgd.aligned_vectors(np.zeros((K, P), np.float32), device)
        self.client_T = [0] * lam
        self.grad_count = [0] * lam
        self.loss_scratch = torch.empty(1024, dtype=torch.float64, device=device)
        self.idx = torch.empty(P, dtype=torch.int32, device=device)
        self.val = torch.empty(P, dtype=torch.float32, device=device)
        self.cnt = torch.empty(1, dtype=torch.int64, device=device)
        self.flag = torch.empty(1, dtype=torch.int32, device=device)
        self.fetched = 0
        self.fetch_opportunities = 0
        # Parameters moved by per-tensor pushes and fetches (device counters).
        self.pushed_params = torch.zeros(1, dtype=torch.int64, device=device)
        self.fetched_params = torch.zeros(1, dtype=torch.int64, device=device)

    def _check(self, rc):
        if rc != fasgd.OK:
            raise fasgd.FasgdError(rc, fasgd.fasgd_last_error(None))

    def loss_into(self, out):
        """f(theta_server) into the device double `out` (no host sync)."""
        self._check(fasgd.fasgd_sim_quadratic_loss(
            self.P, self.srv_theta_ptr(), self.h.data_ptr(), self.star.data_ptr(),
            self.loss_scratch.data_ptr(), out.data_ptr(), self.stream.cuda_stream))

    def srv_theta_ptr(self):
        if not hasattr(self, "_theta_view"):
            self._theta_view = self.torch.empty(self.P, dtype=self.torch.float32, device="cuda")
        self.srv.pull(self._theta_view)
        return self._theta_view.data_ptr()

    def run_batch(self, batch):
        """One dispatcher batch: each client in it pushes a gradient computed on
        its own copy, the server applies the batch, each client refreshes."""
        for k, c in enumerate(batch):
            c = int(c)
            self._check(fasgd.fasgd_sim_quadratic_grad(
                self.P, self.clients[c].data_ptr(), self.h.data_ptr(), self.star.data_ptr(),
                self.sigma.data_ptr(), self.seed, c, self.grad_count[c], self.grads[k].data_ptr(),
                self.stream.cuda_stream))
            self.grad_count[c] += 1
            if self.push_budget is None:
                self.srv.push(c, self.client_T[c], self.grads[k])
            else:
                self.srv.push_budget(c, self.client_T[c], self.grads[k], self.push_budget,
                                     count_dev=self.cnt)
                self.srv.apply_pending(1)
                self.pushed_params += self.cnt
        if self.push_budget is None:
            self.srv.apply_pending(len(batch))
        T = self.srv.T
        for c in batch:
            c = int(c)
            self.fetch_opportunities += 1
            if self.fetch == "full":
                self.srv.pull(self.clients[c])
                self.client_T[c] = T
                self.fetched += 1
            elif self.fetch == "param":
                # The client's parameters become a mix of ages; it reports the
                # timestamp of this fetch (a reading: the paper's timestamps are
                # per message).
                self.srv.fetch_compact(c, self.idx, self.val, self.cnt)
                fasgd.fetch_apply(self.clients[c], self.idx, self.val, n_dev=self.cnt,
                                  n_max=self.P, stream=self.stream)
                self.client_T[c] = T
            elif self.fetch == "budget":
                # As for per-parameter fetches, the client reports this fetch's
                # timestamp.
                self.srv.fetch_budget(c, self.clients[c], self.fetch_budget, count_dev=self.cnt)
                self.fetched_params += self.cnt
                self.client_T[c] = T
            else:
                self.srv.fetch_message(c, self.clients[c], fetched_dev=self.flag)
                if int(self.flag.item()):
                    self.client_T[c] = T
                    self.fetched += 1

    def run(self, schedule, log_every: int = 0):
        """Run every batch of `schedule`; returns the losses logged every
        `log_every` batches (and at the end)."""
        torch = self.torch
        n_log = (len(schedule) // log_every if log_every else 0) + 1
        losses = torch.zeros(n_log, dtype=torch.float64, device="cuda")
        li = 0
        for b, batch in enumerate(schedule):
            self.run_batch(batch)
            if log_every and (b + 1) % log_every == 0 and li < n_log - 1:
                self.loss_into(losses[li:li + 1])
                li += 1
        self.loss_into(losses[li:li + 1])
        return losses[:li + 1].cpu().numpy()

    def close(self):
        self.srv.close()


def compare(P: int, lam: int, n_batches: int, K: int, alphas, seed: int = 0, log_every: int = 0,
            noise: str = "independent"):
    """Final loss of each update rule at each learning rate (same schedule,
    objective and start for all)."""
    sched = streams.dispatch_schedule(seed, lam, n_batches, K)
    obj = streams.quadratic_objective(seed, P, noise=noise)
    th0 = np.zeros(P, np.float32)
    init = float(0.5 * np.sum(obj[0].astype(np.float64) * (th0 - obj[1]).astype(np.float64) ** 2))
    out = {"P": P, "lambda": lam, "K": K, "batches": n_batches, "noise": noise,
           "initial_loss": init, "runs": []}
    for name, var in (("asgd", fasgd.ASGD), ("sasgd", fasgd.SASGD), ("fasgd", fasgd.FASGD),
                      ("fasgd-std", fasgd.FASGD_STD)):
        for a in alphas[name]:
            sim = Simulation(P, lam, a, var, K=K, seed=seed, objective=obj, theta0=th0)
            t0 = time.perf_counter()
            losses = sim.run(sched, log_every)
            el = time.perf_counter() - t0
            sim.close()
            out["runs"].append({"rule": name, "alpha": a, "final_loss": float(losses[-1]),
                                "curve": [float(x) for x in losses], "seconds": el,
                                "pushes_per_s": n_batches * K / el})
    return out


def bandwidth_compare(P: int, lam: int, n_batches: int, T: int, fractions, seed: int = 0,
                      noise: str = "independent"):
    """Per-tensor fetch budgets (the future-work section's allocation by
    statistics) against the same budgets spread uniformly over the tensors
    (eps_b so large that every tensor's Eq. 9 probability is the same) and
    against full fetches: for each rule and each fetch mode, the best final
    loss over a learning-rate sweep, on one schedule, objective and start."""
    sizes = streams.tensor_sizes(seed, P, T)
    sched = streams.dispatch_schedule(seed, lam, n_batches, 1)
    obj = streams.quadratic_objective(seed, P, noise=noise, tensors=sizes)
    th0 = np.zeros(P, np.float32)
    grid = [10.0 ** e for e in np.arange(-5.0, 0.01, 0.5)]
    rules = (("sasgd", fasgd.SASGD, grid), ("fasgd", fasgd.FASGD, grid),
             ("fasgd-std", fasgd.FASGD_STD, [g * 1e-3 for g in grid]))
    modes = [("full", {})]
    for f in fractions:
        modes.append((f"stats_{f}", {"fetch": "budget", "fetch_budget": int(f * P)}))
        modes.append((f"uniform_{f}", {"fetch": "budget", "fetch_budget": int(f * P), "eps_b": 1e6}))
    out = {"P": P, "lambda": lam, "tensors": T, "batches": n_batches, "noise": noise,
           "initial_loss": float(0.5 * np.sum(obj[0].astype(np.float64) * obj[1].astype(np.float64) ** 2)),
           "rows": []}
    for name, var, alphas in rules:
        row = {"rule": name}
        for mode, kw in modes:
            best = (np.inf, None, 0.0)
            for a in alphas:
                sim = Simulation(P, lam, a, var, seed=seed, objective=obj, theta0=th0,
                                 tensor_sizes=sizes, **kw)
                loss = float(sim.run(sched)[-1])
                moved = int(sim.fetched_params.item()) / (n_batches * P)
                sim.close()
                if np.isfinite(loss) and loss < best[0]:
                    best = (loss, a, moved)
            row[mode] = {"loss": best[0], "alpha": best[1], "fetched_fraction": best[2]}
        out["rows"].append(row)
    return out


def main():
    ap = argparse.ArgumentParser(description=__doc__,
                                 formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--compare", action="store_true")
    ap.add_argument("--P", type=int, default=159_010)      # the paper's 784-200-10 MLP size
    ap.add_argument("--lam", type=int, default=128)
    ap.add_argument("--batches", type=int, default=2000)
    ap.add_argument("--K", type=int, default=1)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--noise", choices=["independent", "fisher"], default="independent")
    ap.add_argument("--bandwidth", action="store_true",
                    help="compare per-tensor fetch budgets (by statistics vs uniform)")
    ap.add_argument("--tensors", type=int, default=16)
    args = ap.parse_args()
    if args.bandwidth:
        print(json.dumps(bandwidth_compare(args.P, args.lam, args.batches, args.tensors,
                                           (0.1, 0.3), args.seed, args.noise)))
        return
    grid = [10.0 ** e for e in np.arange(-5.0, 1.01, 0.5)]
    alphas = {"asgd": grid, "sasgd": grid, "fasgd": grid, "fasgd-std": [g * 1e-3 for g in grid]}
    res = compare(args.P, args.lam, args.batches, args.K, alphas, args.seed,
                  log_every=max(1, args.batches // 20), noise=args.noise)
    best = {}
    for r in res["runs"]:
        if np.isfinite(r["final_loss"]) and (r["rule"] not in best or
                                             r["final_loss"] < best[r["rule"]]["final_loss"]):
            best[r["rule"]] = r
    res["best"] = {k: {"alpha": v["alpha"], "final_loss": v["final_loss"],
                       "curve": v["curve"]} for k, v in best.items()}
    summary = {"P": res["P"], "lambda": res["lambda"], "K": res["K"], "noise": res["noise"],
               "batches": res["batches"], "initial_loss": res["initial_loss"], "best": res["best"]}
    print(json.dumps(res if args.compare else summary))


if __name__ == "__main__":
    main()
