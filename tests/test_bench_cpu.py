"""bench.py's host-side roofline arithmetic on CPU: the algorithmic bytes of a decode FFN launch are
every weight byte of the experts the step computes (the routed experts it selected and the shared
experts, which every token uses) plus the activations, and the achieved rate is those bytes over
the measured kernel time."""
import numpy as np
import pytest

import bench
from paper_2609_34077_gb300 import inputs as I

PEAKS = {"hbm": 6787.2, "src": "test"}


def _expected(shape, U, steps, T):
    K, S, d, w = shape.K, shape.n_shared, shape.d, shape.w
    experts = sum(U) + steps * S                      # expert blocks read once per step
    rows = T * (K + S)                                # permuted rows per step
    weights = experts * 3 * w * d * 2                 # W1, W3 and W2 in bf16
    acts = steps * (T * d * 2 + rows * w * 2 + rows * (w * 2 + d * 4))
    return weights + acts


@pytest.mark.parametrize("shape,T,U", [(I.DSV2_LITE, 1, [6, 6, 5]), (I.DSV2_LITE, 64, [50, 48]),
                                       (I.MIXTRAL, 16, [7, 8, 6, 8])],
                         ids=["dsv2-b1", "dsv2-b64", "mixtral-b16"])
def test_decode_roofline_counts_shared_experts(shape, T, U):
    steps = len(U)
    ms = 1.0  # total kernel time of the launches
    prof = {"ffn_decode": (2 * steps, ms)}
    roof, rates = bench.decode_roofline(prof, U, steps, T, shape, PEAKS)
    alg = _expected(shape, U, steps, T)
    assert roof["kernel"] == "ffn_decode"
    assert roof["alg_bytes_per_launch"] == pytest.approx(alg / (2 * steps))
    assert rates["ffn_decode"] == pytest.approx(alg / 1e-3 / 1e9)
    assert roof["frac"] == pytest.approx(rates["ffn_decode"] / PEAKS["hbm"])
    # one DeepSeek token streams 8 expert blocks (6 routed + 2 shared), not 6
    if shape is I.DSV2_LITE and T == 1:
        per_step_weights = roof["alg_bytes_per_launch"] * 2 - (T * shape.d * 2 + 8 * shape.w * 4
                                                                 + 8 * shape.d * 4)
        assert per_step_weights / shape.expert_bytes == pytest.approx((sum(U) / steps) + 2)


def test_traffic_ratio_is_null_for_a_changed_source(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (tmp_path / "k.cu").write_text("kernel source")
    monkeypatch.setitem(bench.TRAFFIC, "k", ("k.cu", "0" * 16, 1.0))
    assert bench.traffic_ratio("k") is None
    import hashlib

    digest = hashlib.sha256(b"kernel source").hexdigest()[:16]
    monkeypatch.setitem(bench.TRAFFIC, "k", ("k.cu", digest, 1.25))
    assert bench.traffic_ratio("k") == 1.25


def test_lora_work_mixtral():
    """Mixtral-shaped T = 4096, rank 8: 8192 permuted rows; the down projections read each 8 KB
    x row and each 28 KB h row once and write 16 + 8 bf16 values; the base GEMMs are 2.886 TFLOP
    and the adapters add 0.25 % (up) on the tensor cores."""
    wk = bench.lora_work(I.MIXTRAL, 4096, 8)
    assert wk["rows"] == 8192
    assert wk["down_bytes"] == 8192 * (4096 * 2 + 32) + 8192 * (14336 * 2 + 16)
    assert wk["base_flop"] == pytest.approx(2.886e12, rel=1e-3)
    assert wk["up_flop"] / wk["base_flop"] == pytest.approx(8 * (2 * 14336 + 4096) / (3 * 4096 * 14336))
    # DeepSeek: the two shared experts are adapted rows too
    assert bench.lora_work(I.DSV2_LITE, 4096, 8)["rows"] == 4096 * 8


def test_gate_grad_bytes():
    """Mixtral-shaped T = 4096: 8192 fp32 rows of 16 KB, 4096 bf16 dL/dy rows of 8 KB, ids and
    gradients: 167.8 MB, the figure the ncu capture reads back."""
    b = bench.gate_grad_bytes(I.MIXTRAL, 4096)
    assert b == 8192 * 4096 * 4 + 4096 * 4096 * 2 + 8192 * 8
    assert b / 1e6 == pytest.approx(167.84, abs=0.01)


def _oracle_ids(shape, batch, seed, n):
    import oracle

    xs = I.ar1_streams(seed, shape, bench.STREAM_STEPS, batch)
    wr = I.router_weight(seed, shape).double().numpy()
    prior = I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep))
    idx = np.zeros((bench.STREAM_STEPS, batch, shape.K), np.int32)
    for p in range(n):
        idx[p] = oracle.routing.route(xs[p].double().numpy(), wr, shape.K,
                                      oracle.routing.MODE_SOFT_PRIOR, shape.gate, prior=prior)["idx"]
    return idx


def test_oracle_fetch_check_counts_and_flags():
    """The bench's fetches-exact check: the oracle's own ids pass with matching counts; a changed
    id outside a near tie is reported, and counts that differ from the replay are not exact."""
    import oracle

    shape, batch, seed, first, steps = I.DSV2_LITE, 2, 5, 4, 12
    idx = _oracle_ids(shape, batch, seed, first + steps)
    chk = bench.oracle_fetch_check(shape, batch, seed, idx, first, steps)
    assert chk["tokens"] == steps * batch and chk["ids_differ_outside_band"] == 0
    assert (chk["oracle_hits"], chk["oracle_fetches"]) == (chk["replay_hits"], chk["replay_fetches"])
    # counts taken independently: a fresh LRU over the same ids
    c = oracle.cache.SlotCache(shape.E, shape.cache_slots, "LRU")
    h = f = 0
    for s in range(first + steps):
        hs, fs, _, _ = c.step(idx[s])
        if s >= first:
            h, f = h + hs, f + fs
    ok = bench.fetch_verdict(chk, h, f)
    assert ok["fetches_exact"] and ok["cache_exact"] and ok["routing_exact_outside_band"]
    assert not bench.fetch_verdict(chk, h, f + 1)["fetches_exact"]
    # plant a different expert for one token of a timed step (not a near tie): flagged
    bad = idx.copy()
    t_pos = first + 3
    row = bad[t_pos, 0]
    row[-1] = next(e for e in range(shape.E) if e not in row)
    chk2 = bench.oracle_fetch_check(shape, batch, seed, bad, first, steps)
    assert chk2["ids_differ_outside_band"] + chk2["ids_differ_in_band"] == 1
    assert not bench.fetch_verdict(chk2, h, f)["routing_exact_outside_band"] or \
        chk2["ids_differ_in_band"] == 1


def test_step_floor_bounds():
    """The step floors: link time of the misses (or the FFN bytes at HBM speed, whichever is
    larger), and that plus the misses' FFN; fractions of the measured step."""
    import bench

    d = dict(ms_per_step=0.150, fetch_bytes_per_step=24.0e6, ffn_dram_bytes_per_step=138.0e6)
    f = bench.step_floor(d, 200.0, 6000.0)
    assert abs(f["link_ms"] - 0.120) < 1e-9
    assert abs(f["link_plus_miss_ffn_ms"] - 0.124) < 1e-9
    assert abs(f["frac_of_link"] - 0.8) < 1e-9
    # no misses: the FFN at HBM speed is the bound
    d0 = dict(ms_per_step=0.030, fetch_bytes_per_step=0.0, ffn_dram_bytes_per_step=138.0e6)
    f0 = bench.step_floor(d0, 200.0, 6000.0)
    assert abs(f0["link_ms"] - 0.023) < 1e-9 and f0["link_ms"] == f0["link_plus_miss_ffn_ms"]


def test_step_floor_per_step_is_tighter():
    """With per-step fetch counts the floor is the mean of each step's own bound: one step that
    fetches and three that only stream their FFN bound the steps more tightly than the averages."""
    import bench

    eb, ffn = 352321536, 704.6e6
    d = dict(ms_per_step=0.5, fetch_bytes_per_step=eb / 4, ffn_dram_bytes_per_step=ffn,
             per_step=dict(fetches=[1, 0, 0, 0], experts=[2] * 4, expert_bytes=eb,
                           ffn_bytes=[ffn] * 4))
    f = bench.step_floor(d, 200.0, 6000.0)
    link = eb / 200e6  # ms for one expert over the link
    hbm = ffn / 6000e6
    assert abs(f["step_ms"] - (link + 3 * hbm) / 4) < 1e-12
    assert abs(f["step_plus_miss_ffn_ms"] - (link + eb / 6000e6 + 3 * hbm) / 4) < 1e-12
    assert f["step_ms"] > f["link_ms"]
