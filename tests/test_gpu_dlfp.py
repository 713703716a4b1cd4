"""The completion-timed DLFP loop on the GPU.

The continuous-batching scheduler (``dlfp.Scheduler``) with the Eq. 2
controller (§3.1) drives the CUDA library through ``Context.iteration``: each
iteration's device-completion time is the L_t the controller observes.
Checked here:

- every guarded cycle's cap follows Eq. 2 from the device time the previous
  guarded cycle returned, replayed with the oracle's restatement of Eq. 2
  and the §3.1 activation/reset rules (``oracle.controller.cycle``);
- every chunk respects its cap and the token budget;
- a sample of the iterations the loop executed matches the float64 oracle
  (layer 0: every decode row and sampled chunk rows, all heads; the KV pages
  the iteration appended, bit-exact).
"""
import numpy as np
import pytest

import oracle
import synth
from oracle import controller as oc
from synth import workload as wl
from tests import harness
from tests.harness import MAX_ABS, MEAN_ABS

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

LAYERS = 4
HQ = 16


class _Engine:
    """Per-layer pools, one row of the page table per request, q/k/v drawn
    afresh for every iteration from the seeded generator; `execute` runs one
    iteration and returns its device time, snapshotting layer 0 around the
    iterations listed in `check_at` for the oracle."""

    def __init__(self, requests, seed, budget, max_seqs, check_at):
        from paper_2609_38386_gb300 import Context
        self.geom = g = wl.Geometry(HQ)
        self.layout = lay = wl.make_layout(g, [r.prompt + r.output for r in requests], seed=seed)
        self.max_tok = budget + max_seqs
        self.ctx = Context(num_q_heads=HQ, num_kv_heads=g.hkv, num_pages=lay.num_pages,
                           num_seqs=lay.num_seqs, max_pages_per_seq=lay.max_pages,
                           max_tokens=self.max_tok, max_decodes=max_seqs)
        self.pt = torch.from_numpy(lay.page_table).cuda()
        self.seed = seed
        self.pools = []
        for l in range(LAYERS):
            kp = synth.fill(synth.stream_base(seed, 100 + 2 * l), lay.pool_shape())
            vp = synth.fill(synth.stream_base(seed, 101 + 2 * l), lay.pool_shape())
            self.pools.append((torch.from_numpy(kp.view(np.int16)).cuda(),
                               torch.from_numpy(vp.view(np.int16)).cuda()))
        self.outs = [torch.empty((self.max_tok, HQ, 128), dtype=torch.int16, device="cuda")
                     for _ in range(LAYERS)]
        self.check_at = set(check_at)
        self.n = 0
        self.checked = []

    def execute(self, plan):
        lay, g = self.layout, self.geom
        nd, p = len(plan.decode_ids), plan.p_t
        n_tok = nd + p
        parts = [lay.slot(rid, c)[None] for rid, c in zip(plan.decode_ids, plan.decode_ctx)]
        if p:
            parts.append(lay.slot(plan.prefill_id, np.arange(plan.chunk_start, plan.chunk_start + p)))
        slots = np.concatenate(parts).astype(np.int32)
        base = lambda s: synth.stream_base(self.seed, 10000 + 3 * self.n + s)
        q = synth.fill(base(0), (n_tok, HQ, 128))
        k = synth.fill(base(1), (n_tok, g.hkv, 128))
        v = synth.fill(base(2), (n_tok, g.hkv, 128))
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()
        d_q, d_k, d_v, d_sl = t(q), t(k), t(v), torch.from_numpy(slots).cuda()
        desc = self.ctx.make_desc(decode_seq_ids=plan.decode_ids, decode_ctx_lens=plan.decode_ctx,
                                  prefill_seq_id=plan.prefill_id, chunk_start=plan.chunk_start,
                                  p_t=p, page_table=self.pt, slots=d_sl)
        snap = None
        if self.n in self.check_at:
            snap = (self.pools[0][0].cpu().numpy().view(np.uint16).copy(),
                    self.pools[0][1].cpu().numpy().view(np.uint16).copy())
        layers = [self.ctx.make_bufs(d_q, d_k, d_v, kp, vp, o) for (kp, vp), o in zip(self.pools, self.outs)]
        us = self.ctx.iteration(desc, layers)
        if snap is not None:
            self._check(plan, q, k, v, slots, snap, n_tok)
        self.n += 1
        return us

    def _check(self, plan, q, k, v, slots, snap, n_tok):
        nd, p = len(plan.decode_ids), plan.p_t
        kp, vp = snap
        rows = list(range(nd))
        if p:
            rng = np.random.default_rng(self.n)
            rows += sorted({nd, nd + p - 1} | {int(x) for x in rng.integers(nd, n_tok, size=min(p, 30))})
        want, _ = oracle.mixed_attention(
            q=q, k=k, v=v, k_pool=kp, v_pool=vp, page_table=self.layout.page_table, slots=slots,
            decode_seq_ids=np.asarray(plan.decode_ids, np.int32),
            decode_ctx_lens=np.asarray(plan.decode_ctx, np.int32),
            prefill_seq=plan.prefill_id, chunk_start=plan.chunk_start, p_t=p, rows=rows)
        got = harness._bf16_to_f64(self.outs[0][:n_tok].cpu().numpy()[rows])
        assert np.all(np.isfinite(got))
        err = np.abs(got - want)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (self.n, err.max(), err.mean())
        # kp/vp now hold the oracle's append: the device pools must equal them
        np.testing.assert_array_equal(self.pools[0][0].cpu().numpy().view(np.uint16), kp)
        np.testing.assert_array_equal(self.pools[0][1].cpu().numpy().view(np.uint16), vp)
        self.checked.append(self.n)


def test_dlfp_loop_on_device_times():
    from paper_2609_38386_gb300 import dlfp
    # a short trace: early requests decode while a long prompt is prefilled
    reqs = [dlfp.Request(0, 0.0, 700, 40), dlfp.Request(1, 0.0, 1500, 40),
            dlfp.Request(2, 1.0, 9000, 8), dlfp.Request(3, 2.0, 5000, 8)]
    budget, max_seqs, n_iter = 8192, 16, 24
    eng = _Engine(reqs, seed=9, budget=budget, max_seqs=max_seqs, check_at=[1, 5, 9, 14])
    # target (us): about the device time of a guarded 4-layer iteration of
    # this workload, so that the cap moves
    target = 150.0
    ctl = dlfp.DLFPController(target)
    sch = dlfp.Scheduler([dlfp.Request(r.rid, r.arrival, r.prompt, r.output) for r in reqs], ctl,
                         max_seqs=max_seqs, budget=budget)
    sch.run(eng.execute, max_iterations=n_iter)
    assert len(sch.log) == n_iter
    assert eng.checked == [1, 5, 9, 14]

    # replay the §3.1 policy on the returned device times
    c = oc.PAPER_C_INIT
    guarded = 0
    for plan, us in sch.log:
        assert us > 0
        nd = len(plan.decode_ids)
        assert nd + plan.p_t <= budget
        # a cycle is guarded (capped) exactly when a decoder is active and a
        # prefill shares it; only a guarded cycle that prefilled feeds back
        cap, c_next = oc.cycle(c, nd, plan.cap is not None, us if plan.p_t else None, target=target)
        if nd == 0:
            assert plan.cap is None and c_next == oc.PAPER_C_INIT
        if plan.cap is not None:
            guarded += 1
            assert plan.cap == cap == c, (plan, c)
            assert plan.p_t <= plan.cap
        c = c_next
    assert guarded >= 5
    assert ctl.updates == guarded
    assert ctl.cap == c
    # the controller moved: the device times drove more than one cap
    caps = {p.cap for p, _ in sch.log if p.cap is not None}
    assert len(caps) >= 2, caps
