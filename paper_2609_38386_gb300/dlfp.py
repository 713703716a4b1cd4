"""Completion-timed Decode-Latency Feedback Prefill (DLFP) scheduling loop.

The paper's controller (§3.1) caps the prefill chunk of each mixed
iteration from an observed iteration latency:

    c_{t+1} = clamp(floor_128(c_t * T / L_t), c_min, c_max)        (Eq. 2)

applied only when at least one request is decoding and a prefill shares the
cycle; with no decoder the cap resets to c_initial and prefill is uncapped.
The paper observed L_t as the host scheduler-call interval and traced its
failures to that proxy (§6.4); §7 and §9 name the fix, a completion-timed
signal.  Here L_t is the device-completion time of the iteration returned by
``Context.iteration`` (CUDA events around the iteration's launches).

``Scheduler`` is a host-side continuous-batching iteration builder in the
vLLM style the paper modifies (§3.2, §4.1): at most ``max_seqs`` running
sequences, a ``budget`` of tokens per iteration shared by the decodes (one
token each) and at most one prefill chunk, prompts admitted in arrival order.
It is independent of the GPU: it calls ``execute(plan) -> device_us`` for
each iteration, so the loop can run against the CUDA library or a model.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

# §3.1: evaluated parameters (T in ms for the paper's whole-model iteration).
PAPER_T_MS = 80.0
C_INIT, C_MIN, C_MAX, QUANTUM = 3072, 1024, 6144, 128


class DLFPController:
    """Eq. 2 with the §3.1 activation and reset rules."""

    def __init__(self, target, c_init=C_INIT, c_min=C_MIN, c_max=C_MAX, quantum=QUANTUM):
        if target <= 0:
            raise ValueError("target latency must be positive")
        self.target = float(target)
        self.c_init, self.c_min, self.c_max, self.quantum = c_init, c_min, c_max, quantum
        self.cap = c_init
        self.updates = 0

    def cap_for(self, n_decoding: int, prefill_pending: bool):
        """Cap for the next cycle: None (uncapped) unless it is guarded."""
        if n_decoding == 0:
            self.cap = self.c_init            # no decoder: reset, prefill free
            return None
        if not prefill_pending:
            return None
        return self.cap

    def observe(self, latency: float):
        """Feed back the completed latency of a guarded cycle."""
        if latency <= 0:
            raise ValueError("latency must be positive")
        q = self.quantum
        nxt = q * math.floor(self.cap * self.target / latency / q)
        self.cap = min(max(nxt, self.c_min), self.c_max)
        self.updates += 1
        return self.cap


class FixedCap:
    """A fixed chunk cap (the paper's fixed-cap controls, §5.3)."""

    def __init__(self, cap):
        self.cap = cap
        self.updates = 0

    def cap_for(self, n_decoding, prefill_pending):
        return self.cap if prefill_pending else None

    def observe(self, latency):
        return self.cap


@dataclasses.dataclass
class Request:
    rid: int
    arrival: float          # same time unit as the device times
    prompt: int
    output: int
    prefilled: int = 0
    generated: int = 0
    first_token: float = -1.0
    finished: float = -1.0
    token_times: list = dataclasses.field(default_factory=list)

    @property
    def ctx(self) -> int:
        """Tokens cached before this iteration's decode token."""
        return self.prompt + self.generated - 1


@dataclasses.dataclass
class TraceSpec:
    """Seeded open-loop trace shaped like the paper's (§4.2): Poisson arrivals,
    lognormal prompt lengths (median 1024, sigma 1, clipped to [64, 16384]),
    output lengths uniform in [64, 512]."""
    n_requests: int = 100
    mean_interarrival: float = 1.0
    prompt_median: int = 1024
    prompt_sigma: float = 1.0
    prompt_min: int = 64
    prompt_max: int = 16384
    out_min: int = 64
    out_max: int = 512
    seed: int = 801

    def requests(self):
        rng = np.random.default_rng(self.seed)
        gaps = rng.exponential(self.mean_interarrival, size=self.n_requests)
        arrivals = np.cumsum(gaps) - gaps[0]
        prompts = np.exp(rng.normal(math.log(self.prompt_median), self.prompt_sigma,
                                    size=self.n_requests))
        prompts = np.clip(np.round(prompts), self.prompt_min, self.prompt_max).astype(int)
        outs = rng.integers(self.out_min, self.out_max + 1, size=self.n_requests)
        return [Request(i, float(a), int(p), int(o))
                for i, (a, p, o) in enumerate(zip(arrivals, prompts, outs))]


@dataclasses.dataclass
class IterationPlan:
    """What one mixed iteration runs (the mx_iter_desc contents)."""
    decode_ids: list            # request ids decoding this iteration
    decode_ctx: list            # their cached lengths
    prefill_id: int             # request id being prefilled, or -1
    chunk_start: int
    p_t: int
    cap: int | None             # the cap that applied (None: uncapped)


class Scheduler:
    """Continuous batching with at most one prefill chunk per iteration."""

    def __init__(self, requests, controller, max_seqs=64, budget=8192):
        self.pending = sorted(requests, key=lambda r: r.arrival)
        self.controller = controller
        self.max_seqs, self.budget = max_seqs, budget
        self.running: list[Request] = []   # admitted, not finished (arrival order)
        self.done: list[Request] = []
        self.clock = 0.0
        self.log = []                      # per iteration: (plan, device_us)

    def _admit(self):
        while (self.pending and self.pending[0].arrival <= self.clock
               and len(self.running) < self.max_seqs):
            self.running.append(self.pending.pop(0))

    def next_plan(self) -> IterationPlan | None:
        self._admit()
        if not self.running:
            if not self.pending:
                return None
            self.clock = max(self.clock, self.pending[0].arrival)   # idle until next arrival
            self._admit()
        decoders = [r for r in self.running if r.prefilled == r.prompt]
        filling = [r for r in self.running if r.prefilled < r.prompt]
        pre = filling[0] if filling else None
        cap = self.controller.cap_for(len(decoders), pre is not None)
        p_t = 0
        if pre is not None:
            room = self.budget - len(decoders)
            p_t = min(pre.prompt - pre.prefilled, room)
            if cap is not None:
                p_t = min(p_t, cap)
            p_t = max(p_t, 0)
        return IterationPlan([r.rid for r in decoders], [r.ctx for r in decoders],
                             pre.rid if (pre is not None and p_t > 0) else -1,
                             pre.prefilled if pre is not None else 0, p_t, cap)

    def commit(self, plan: IterationPlan, device_us: float):
        """Advance the virtual clock by the completed iteration time and apply
        its effects (decode tokens, prefill progress, first tokens)."""
        self.clock += device_us
        self.log.append((plan, device_us))
        by_id = {r.rid: r for r in self.running}
        for rid in plan.decode_ids:
            r = by_id[rid]
            r.generated += 1
            r.token_times.append(self.clock)
        if plan.p_t:
            r = by_id[plan.prefill_id]
            r.prefilled += plan.p_t
            if r.prefilled == r.prompt:         # the prompt's last chunk yields token 1
                r.generated = 1
                r.first_token = self.clock
                r.token_times.append(self.clock)
        if plan.cap is not None and plan.decode_ids and plan.p_t:
            self.controller.observe(device_us)   # guarded cycle: completion-timed feedback
        still = []
        for r in self.running:
            if r.prefilled == r.prompt and r.generated >= r.output:
                r.finished = self.clock
                self.done.append(r)
            else:
                still.append(r)
        self.running = still

    def run(self, execute, max_iterations=10 ** 6):
        for _ in range(max_iterations):
            plan = self.next_plan()
            if plan is None:
                break
            self.commit(plan, float(execute(plan)))
        return self.summary()

    def summary(self):
        it_us = np.array([us for _, us in self.log])
        dec_us = np.array([us for p, us in self.log if p.decode_ids])
        itl = np.concatenate([np.diff(r.token_times) for r in self.done
                              if len(r.token_times) > 1] or [np.zeros(0)])
        ttft = np.array([r.first_token - r.arrival for r in self.done])
        pct = lambda a, q: float(np.percentile(a, q)) if a.size else None
        return {"iterations": int(it_us.size), "requests_done": len(self.done),
                "iter_us_p50": pct(it_us, 50), "iter_us_p99": pct(it_us, 99),
                "decode_iter_us_p50": pct(dec_us, 50), "decode_iter_us_p99": pct(dec_us, 99),
                "itl_p50": pct(itl, 50), "itl_p99": pct(itl, 99),
                "ttft_p50": pct(ttft, 50), "ttft_p99": pct(ttft, 99),
                "makespan": float(self.clock), "controller_updates": self.controller.updates}
