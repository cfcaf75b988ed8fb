"""The attention step on its own (spd_attention, Sec. 3.2 VSkip-Attn: queries are the active tokens,
keys and values every token of the query's sequence) against the oracle's causal attention on the
same bf16 inputs.

Tolerance: output rows within 2e-2 normwise (max_j |gpu - oracle| / max_j |oracle|): the kernel
rounds the softmax weights P and the output to bf16 and accumulates in fp32."""
import numpy as np
import pytest
import torch

from oracle import decoder as od
from paper_2609_34977_gb300 import _native as N
from tests.gpu_util import bf16_np, rowwise_rel

pytestmark = pytest.mark.gpu
TOL = 2e-2


def case(lens, n_heads, n_kv_heads, hd, active_frac, seed, ramp=0.0):
    """Packed sequences of the given lengths; a seeded subset of each sequence's tokens are the
    queries. ramp > 0 makes scores grow along the sequence (each key block raises the running
    maximum, so the output rescaling runs on every block)."""
    r = np.random.default_rng(seed)
    T = sum(lens)
    qd, kvd = n_heads * hd, n_kv_heads * hd
    q_all = r.standard_normal((T, qd))
    k = r.standard_normal((T, kvd))
    v = r.standard_normal((T, kvd))
    pos = np.concatenate([np.arange(n) for n in lens])
    if ramp:
        u = r.standard_normal(hd)
        u /= np.linalg.norm(u)
        q_all += 4.0 * np.tile(u, n_heads)[None, :]
        k += ramp * (pos / max(lens))[:, None] * np.tile(u, n_kv_heads)[None, :]
    q_rows, q_cu = [], [0]
    start = 0
    fracs = active_frac if isinstance(active_frac, list) else [active_frac] * len(lens)
    for n, fr in zip(lens, fracs):
        sel = np.flatnonzero(r.random(n) < fr)
        q_rows.append(start + sel)
        q_cu.append(q_cu[-1] + len(sel))
        start += n
    q_rows = np.concatenate(q_rows).astype(np.int64)
    bf = lambda a: torch.from_numpy(a).float().to(torch.bfloat16)
    q = bf(q_all[q_rows])
    kv = bf(np.concatenate([k, v], axis=1))
    q_pos = pos[q_rows].astype(np.int32)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    return q, q_pos, np.array(q_cu, np.int32), kv, cu


def oracle_attention(q, q_pos, q_cu, kv, cu, n_heads, n_kv_heads, hd):
    qn, kvn = bf16_np(q), bf16_np(kv)
    kvd = n_kv_heads * hd
    out = np.zeros_like(qn)
    for b in range(len(cu) - 1):
        a0, a1, t0, t1 = q_cu[b], q_cu[b + 1], cu[b], cu[b + 1]
        if a1 == a0:
            continue
        out[a0:a1] = od.causal_attention(qn[a0:a1], kvn[t0:t1, :kvd], kvn[t0:t1, kvd:], q_pos[a0:a1],
                                         np.arange(t1 - t0), n_heads, n_kv_heads, hd)
    return out


def run(q, q_pos, q_cu, kv, cu, n_heads, n_kv_heads, hd):
    o = torch.full(tuple(q.shape), float("nan"), dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(N.spd_attention_workspace_size(int(q_cu[-1]), len(cu) - 1), dtype=torch.uint8,
                     device="cuda")
    N.spd_attention(q.cuda(), torch.from_numpy(q_pos).cuda(), q_cu, kv.cuda(), cu, n_heads, n_kv_heads,
                    hd, o, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    return bf16_np(o)


@pytest.mark.parametrize("lens,H,Hkv,hd,frac", [
    ([300, 77, 130], 8, 2, 128, 0.7),    # GQA, ragged sequences, partial key blocks
    ([640], 4, 4, 64, 1.0),              # every token a query: 5 query tiles x 5 key blocks
    ([128, 129, 1, 256], 4, 1, 128, 0.5),  # tile-edge lengths, a one-token sequence
    ([200, 50, 90], 2, 2, 128, [0.5, 0.0, 0.3]),  # a sequence without queries (keys only)
])
def test_attention_matches_oracle(lens, H, Hkv, hd, frac):
    q, q_pos, q_cu, kv, cu = case(lens, H, Hkv, hd, frac, seed=sum(lens) + H)
    got = run(q, q_pos, q_cu, kv, cu, H, Hkv, hd)
    ref = oracle_attention(q, q_pos, q_cu, kv, cu, H, Hkv, hd)
    assert np.isfinite(got).all()
    assert rowwise_rel(got, ref) < TOL


def test_attention_running_maximum_rescales_every_block():
    q, q_pos, q_cu, kv, cu = case([512, 384], 4, 2, 128, 0.8, seed=11, ramp=12.0)
    got = run(q, q_pos, q_cu, kv, cu, 4, 2, 128)
    ref = oracle_attention(q, q_pos, q_cu, kv, cu, 4, 2, 128)
    assert rowwise_rel(got, ref) < TOL


def test_attention_first_key_only():
    # the query at position 0 sees only itself: its output is exactly V of token 0 (up to bf16)
    q, q_pos, q_cu, kv, cu = case([1, 1, 1], 2, 2, 64, 1.0, seed=3)
    got = run(q, q_pos, q_cu, kv, cu, 2, 2, 64)
    np.testing.assert_allclose(got, bf16_np(kv)[:, 128:], rtol=1e-2, atol=1e-2)
