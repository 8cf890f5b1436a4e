"""Closed-loop simulation on the CPU oracle -- TEST INFRASTRUCTURE ONLY.

The same protocol as paper_1601_04033_gb300.sim (dispatcher schedule from
streams.dispatch_schedule, clients computing gradients of the synthetic
quadratic at their own copies, the server applying each batch, clients
refreshing), with the oracle's server, gradient and loss.
"""

from __future__ import annotations

import numpy as np

from . import OracleServer, fetch_apply, sim_grad, sim_loss


class OracleSimulation:
    def __init__(self, P, lam, alpha, variant, *, gamma=0.95, beta=0.95, eps=1e-4, seed=0,
                 fetch="full", c_fetch=0.0, objective, theta0, lib=None, eps_b=1e-8,
                 tensor_sizes=None, fetch_budget=None, push_budget=None):
        self.P, self.lam, self.seed, self.fetch = P, lam, seed, fetch
        self.lib = lib
        self.srv = OracleServer(P, lam, alpha, variant, gamma=gamma, beta=beta, eps=eps, seed=seed,
                                eps_b=eps_b, lib=lib)
        if tensor_sizes is not None:
            self.srv.set_tensors(tensor_sizes)
        self.fetch_budget, self.push_budget = fetch_budget, push_budget
        self.srv.set_fetch_threshold(c_fetch)
        self.srv.set_params(theta0)
        self.h, self.star, self.sigma = [np.ascontiguousarray(x, np.float32) for x in objective]
        self.clients = [np.array(theta0, dtype=np.float32) for _ in range(lam)]
        self.client_T = [0] * lam
        self.grad_count = [0] * lam

    def loss(self):
        return sim_loss(self.srv.theta.astype(np.float32), self.h, self.star, lib=self.lib)

    def run_batch(self, batch):
        for c in batch:
            c = int(c)
            g = sim_grad(self.clients[c], self.h, self.star, self.sigma, self.seed, c,
                         self.grad_count[c], lib=self.lib)
            self.grad_count[c] += 1
            if self.push_budget is None:
                self.srv.push(c, self.client_T[c], g)
            else:
                self.srv.push_budget(c, self.client_T[c], g, self.push_budget)
                self.srv.apply_pending(1)
        if self.push_budget is None:
            self.srv.apply_pending(len(batch))
        T = self.srv.T
        for c in batch:
            c = int(c)
            if self.fetch == "full":
                self.clients[c][:] = self.srv.theta.astype(np.float32)
                self.client_T[c] = T
            elif self.fetch == "param":
                idx, val = self.srv.fetch_compact(c)
                fetch_apply(self.clients[c], idx, val, lib=self.lib)
                self.client_T[c] = T
            elif self.fetch == "budget":
                self.srv.fetch_budget(c, self.clients[c], self.fetch_budget)
                self.client_T[c] = T
            else:
                if self.srv.fetch_message(c, self.clients[c]):
                    self.client_T[c] = T

    def run(self, schedule, log_every=0):
        out = []
        for b, batch in enumerate(schedule):
            self.run_batch(batch)
            if log_every and (b + 1) % log_every == 0:
                out.append(self.loss())
        out.append(self.loss())
        return np.array(out)
