"""bench.py's host-side roofline arithmetic on CPU: the algorithmic bytes of a decode FFN launch are
every weight byte of the experts the step computes (the routed experts it selected and the shared
experts, which every token uses) plus the activations, and the achieved rate is those bytes over
the measured kernel time."""
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
    monkeypatch.setitem(bench.TRAFFIC, "k", ("k.cu", "0" * 16, 1.0, "profiles/k.md"))
    assert bench.traffic_ratio("k") is None
    import hashlib

    digest = hashlib.sha256(b"kernel source").hexdigest()[:16]
    monkeypatch.setitem(bench.TRAFFIC, "k", ("k.cu", digest, 1.25, "profiles/k.md"))
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
