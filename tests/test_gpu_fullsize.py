"""Parity at full workload sizes, in the launch configuration the bench uses
(its planner, grid and split heuristics): every decode row and the first,
last and 62 random rows of the chunk, all heads, against the float64 oracle
on the pages those rows read; plus every appended page bit-exact and a
sample of untouched pages unchanged.

Workloads: the Qwen3-0.6B 28-layer sweep (one layer call of selected
iterations), and the Qwen3-8B / 32B attention geometries (32 / 64 query
heads, 64 / 128 decodes with log-uniform contexts up to 8K / 16K, prompts of
16K / 32K tokens).
"""
import numpy as np
import pytest

from synth import workload as wl
from tests import harness
from tests.harness import MAX_ABS, MEAN_ABS, Case

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _pick(cfg, chunk, which):
    its = [i for i, it in enumerate(cfg.iterations()) if it.chunk_size == chunk]
    return its[0] if which == "first" else its[-1]


CASES = [
    ("qwen3-0.6b-attn-28L-chunk-sweep", 0, "first"),
    ("qwen3-0.6b-attn-28L-chunk-sweep", 256, "last"),     # key-split prefill pieces
    ("qwen3-0.6b-attn-28L-chunk-sweep", 2048, "last"),
    ("qwen3-0.6b-attn-28L-chunk-sweep", 4096, "first"),
    ("qwen3-8b-attn-36L-chunk-sweep", 512, "last"),
    ("qwen3-8b-attn-36L-chunk-sweep", 4096, "first"),
    ("qwen3-32b-attn-64L-chunk-sweep", 0, "first"),
    ("qwen3-32b-attn-64L-chunk-sweep", 1024, "last"),
    ("qwen3-32b-attn-64L-chunk-sweep", 8192, "last"),     # deepest items the bench times
]


@pytest.mark.parametrize("name,chunk,which", CASES)
def test_fullsize_sampled_parity(name, chunk, which):
    cfg = wl.CONFIGS[name]
    case = Case.from_config(cfg, _pick(cfg, chunk, which), layer=3, device_pools=True)
    res = case.run_gpu(keep=True)
    rows = case.sample_rows(62, seed=chunk)
    err = harness.compare_rows(case, res, rows)
    assert err["max_abs"] <= MAX_ABS and err["mean_abs"] <= MEAN_ABS, err
    assert harness.check_pages(case, res["dev"]) > 0
    # rows the oracle did not sample are written and finite
    out = harness._bf16_to_f64(res["out"])
    assert np.all(np.isfinite(out))
    res["ctx"].close()
