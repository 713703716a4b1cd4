"""KV-head sharding of the mixed attention across GPUs (tensor parallelism of
attention, the paper's two-GPU setting, §4.1 / §5).

Attention of one KV head touches only that head's pages and the query heads
of its group (query head h reads KV head h / (Hq / Hkv)), so a rank that holds
KV heads [a, b) and query heads [a n_rep, b n_rep) runs the unchanged
single-GPU launch on its share with no exchange inside attention: its
context has b - a KV heads, its pools [pages][b - a][16][128] hold only those
heads, its q/k/v/out only those heads' columns.  The heads' outputs are
joined after attention (by the output projection's reduction in a model).
"""
from __future__ import annotations


def kv_head_range(num_kv_heads, rank, world):
    """KV heads [a, b) of `rank`: contiguous, as equal as the count allows."""
    if not (0 <= rank < world) or world > num_kv_heads:
        raise ValueError("need 0 <= rank < world <= num_kv_heads")
    a = rank * num_kv_heads // world
    b = (rank + 1) * num_kv_heads // world
    return a, b


def shard_geometry(num_q_heads, num_kv_heads, rank, world):
    """(q heads [qa, qb), kv heads [a, b)) of `rank`: each KV head with its
    whole query group."""
    if num_q_heads % num_kv_heads:
        raise ValueError("num_q_heads must be a multiple of num_kv_heads")
    n_rep = num_q_heads // num_kv_heads
    a, b = kv_head_range(num_kv_heads, rank, world)
    return (a * n_rep, b * n_rep), (a, b)


def take_heads(t, heads, dim):
    """The contiguous copy of heads [h0, h1) of tensor t along dim `dim`."""
    h0, h1 = heads
    return t.narrow(dim, h0, h1 - h0).contiguous()
