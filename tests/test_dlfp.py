"""DLFP controller and scheduling loop (host logic, no GPU).

The product controller is checked against the oracle's restatement of §3.1
Eq. 2 and the paper's worked example; the scheduler against the invariants
of continuous batching with one prefill chunk per iteration (§2.1, §3.2,
§4.1 budget and sequence limits), driven by a deterministic iteration-time
model instead of the GPU.
"""
import os

import numpy as np
import pytest

from oracle import controller as oc
from paper_2609_38386_gb300 import dlfp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "dlfp_controller_example.txt")


def test_worked_example_from_the_paper():
    line = [l for l in open(GOLDEN) if l.strip() and not l.startswith("#")][0]
    g = {k: float(v) for k, v in (t.split("=") for t in line.split())}
    c = dlfp.DLFPController(target=g["T_ms"])
    c.cap = int(g["c_t"])
    assert c.cap_for(n_decoding=4, prefill_pending=True) == 3072
    assert c.observe(g["observed_ms"]) == int(g["c_next"]) == 4224


def test_controller_matches_oracle_restatement():
    rng = np.random.default_rng(0)
    c = dlfp.DLFPController(target=80.0)
    cap = oc.PAPER_C_INIT
    for _ in range(2000):
        nd = int(rng.integers(0, 4))
        pending = bool(rng.integers(0, 2))
        obs = float(rng.uniform(5, 400))
        applied, cap_next = oc.cycle(cap, nd, pending, obs)
        got = c.cap_for(nd, pending)
        assert got == applied
        if applied is not None:
            c.observe(obs)
        assert c.cap == cap_next
        cap = cap_next


def _model(plan):
    # a deterministic latency model: decode bytes + prefill flops + overhead
    dec = sum(plan.decode_ctx) * 0.01
    pre = plan.p_t * (plan.chunk_start + plan.p_t / 2) * 2e-5 + plan.p_t * 0.05
    return 50.0 + dec + pre


@pytest.mark.parametrize("policy", ["dlfp", "fixed"])
def test_scheduler_invariants(policy):
    spec = dlfp.TraceSpec(n_requests=40, mean_interarrival=400.0, seed=801)
    reqs = spec.requests()
    ctl = dlfp.DLFPController(target=300.0) if policy == "dlfp" else dlfp.FixedCap(2048)
    sch = dlfp.Scheduler(reqs, ctl, max_seqs=16, budget=4096)
    prefilled = {r.rid: 0 for r in reqs}
    decoded = {r.rid: 0 for r in reqs}

    def execute(plan):
        assert len(plan.decode_ids) <= 16
        assert len(plan.decode_ids) + plan.p_t <= 4096
        if plan.cap is not None:
            assert plan.p_t <= plan.cap
            if policy == "dlfp":
                assert plan.decode_ids, "DLFP caps only prefills beside active decodes"
        if plan.p_t:
            assert prefilled[plan.prefill_id] == plan.chunk_start   # chunks in order
            prefilled[plan.prefill_id] += plan.p_t
        for rid, ctx in zip(plan.decode_ids, plan.decode_ctx):
            r = reqs[rid]
            assert prefilled[rid] == r.prompt                       # decode after prefill
            assert ctx == r.prompt + decoded[rid]                   # cache grows by one
            decoded[rid] += 1
        return _model(plan)

    out = sch.run(execute)
    assert out["requests_done"] == 40
    for r in reqs:
        assert prefilled[r.rid] == r.prompt
        assert decoded[r.rid] == r.output - 1       # token 1 comes from the prefill
        assert len(r.token_times) == r.output
        assert r.first_token >= r.arrival
        assert np.all(np.diff(r.token_times) > 0)
    if policy == "dlfp":
        assert out["controller_updates"] > 0
        assert dlfp.C_MIN <= ctl.cap <= dlfp.C_MAX and ctl.cap % dlfp.QUANTUM == 0


def test_dlfp_reduces_tail_iteration_time_under_the_model():
    """With latency growing in the chunk size, capping chunks beside decodes
    lowers the tail of decode-carrying iteration times (the §5.1 effect)."""
    spec = dlfp.TraceSpec(n_requests=60, mean_interarrival=2000.0, prompt_median=4096,
                          seed=802)
    res = {}
    for name, ctl in [("fixed", dlfp.FixedCap(8192)),
                      ("dlfp", dlfp.DLFPController(target=600.0, c_init=2048,
                                                   c_min=256, c_max=8192))]:
        sch = dlfp.Scheduler(spec.requests(), ctl, max_seqs=32, budget=8192)
        res[name] = sch.run(_model)
    assert res["dlfp"]["decode_iter_us_p99"] < res["fixed"]["decode_iter_us_p99"]
    assert res["dlfp"]["requests_done"] == res["fixed"]["requests_done"] == 60


def test_trace_is_seeded_and_shaped():
    a = dlfp.TraceSpec(seed=801).requests()
    b = dlfp.TraceSpec(seed=801).requests()
    assert [(r.arrival, r.prompt, r.output) for r in a] == [(r.arrival, r.prompt, r.output) for r in b]
    p = np.array([r.prompt for r in a])
    o = np.array([r.output for r in a])
    assert p.min() >= 64 and p.max() <= 16384 and o.min() >= 64 and o.max() <= 512
    assert 500 < np.median(p) < 2000
