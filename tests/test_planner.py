"""The library's work planners, checked on the CPU (no GPU needed) through
simsd_plan_attention / simsd_plan_accept, which take the SM count as an
argument: the plans equal the rules restated in tests/_plan.py over a grid
of shapes and SM counts, the decisions the measurements rest on hold
(stream-K for long 256-row units that load the SMs unevenly, whole units
for short ones, ranges for small batches, the split acceptance passes of
few sequences in one wave), and bad arguments are rejected."""
import itertools

import pytest

from tests import _plan

SMS = (132, 148, 152, 160)


@pytest.fixture(scope="module")
def simsd():
    from paper_2606_02544_gb300 import build, simsd
    build.build()
    return simsd


@pytest.mark.parametrize("sms", SMS)
def test_attention_plans_match_the_rules(simsd, sms):
    shapes = itertools.product((1, 2, 5, 8, 18, 19, 20, 24, 32, 40, 64, 128, 255, 256, 300),
                               (0, 100, 512, 2048, 8192, 32768), (16, 64, 256))
    n = 0
    for Bt, keys, P in shapes:
        max_pages = -(-max(keys, 1) // P)
        for gamma, Hq, Hkv in ((32, 32, 8), (16, 32, 8), (4, 16, 8), (8, 32, 8), (16, 64, 8), (20, 32, 8)):
            got = simsd.simsd_plan_attention(simsd.SIMSD_BF16, Bt, gamma, Hq, Hkv, 128, max_pages, P, sms)
            want = _plan.plan_attention(Bt, gamma, Hq, Hkv, max_pages, P, sms)
            assert got == want, (Bt, keys, P, gamma, Hq, Hkv, sms, got, want)
            n += 1
    assert n == 15 * 6 * 3 * 6


def _p(simsd, Bt, keys, sms=152, gamma=32, Hq=32, Hkv=8, P=64):
    return simsd.simsd_plan_attention(simsd.SIMSD_BF16, Bt, gamma, Hq, Hkv, 128, -(-keys // P), P, sms)


def test_attention_decisions(simsd):
    # 256-row units (32 drafts, 32/8 heads)
    assert _p(simsd, 32, 8192)["streamk"] == 1          # 256 units of 129 tiles on 152 SMs: runs
    assert _p(simsd, 32, 32768)["streamk"] == 1
    assert _p(simsd, 64, 8192)["streamk"] == 1
    for keys in (512, 2048):                            # short units: whole
        p = _p(simsd, 32, keys)
        assert p["kernel"] == 1 and p["nsplit"] == 1 and p["streamk"] == 0 and p["ws_bytes"] == 0
    p = _p(simsd, 19, 8192)                             # one unit per SM: whole
    assert p["nsplit"] == 1 and p["streamk"] == 0
    assert _p(simsd, 128, 8192)["streamk"] == 0          # 1024 units: nearly even
    assert _p(simsd, 300, 32768)["streamk"] == 0         # beyond 255 sequences
    assert _p(simsd, 8, 32768)["streamk"] == 1           # 64 units: runs beat ranges
    p = _p(simsd, 8, 8192)                              # ranges beat runs
    assert p["streamk"] == 0 and p["nsplit"] > 1 and p["ws_bytes"] > 0
    p = _p(simsd, 1, 32768)
    assert p["streamk"] == 0 and p["nsplit"] > 1
    assert _p(simsd, 8, 512)["kernel"] == 0              # short units: the one-row-block kernel
    p = _p(simsd, 32, 8192)
    assert p["ws_bytes"] == 152 * (4 * 128 * 130 * 4 + 16)
    # one row block (16 drafts): the SDAR-8B step keeps whole units
    p = _p(simsd, 64, 8192, gamma=16)
    assert p == dict(kernel=0, nsplit=1, streamk=0, rows_blk=128, fuse=0, ws_bytes=0)
    # few units: prefix splits merged in a cluster (2..8), beyond 8 through the workspace
    p = _p(simsd, 8, 1024, gamma=4, Hq=16)
    assert p["fuse"] == 1 and 2 <= p["nsplit"] <= 8 and p["ws_bytes"] == 0
    p = _p(simsd, 1, 8192, gamma=8)
    assert p["fuse"] == 0 and p["nsplit"] > 8 and p["ws_bytes"] > 0


def test_attention_fp32_and_rejections(simsd):
    p = simsd.simsd_plan_attention(simsd.SIMSD_F32, 1, 4, 2, 1, 64, 2, 64, 152)
    assert p["kernel"] == 2 and p["ws_bytes"] == 0
    assert simsd.simsd_plan_attention(simsd.SIMSD_BF16, 0, 32, 32, 8, 128, 10, 64, 152)["ws_bytes"] == 0
    bad = [(simsd.SIMSD_BF16, 4, 0, 32, 8, 128, 10, 64, 152),      # gamma 0
           (simsd.SIMSD_BF16, 4, 33, 32, 8, 128, 10, 64, 152),     # gamma 33
           (simsd.SIMSD_BF16, 4, 4, 30, 8, 128, 10, 64, 152),      # Hq not a multiple of Hkv
           (simsd.SIMSD_BF16, 4, 4, 32, 8, 128, 10, 64, 0)]        # no SMs
    for args in bad:
        with pytest.raises(simsd.SimsdError) as exc:
            simsd.simsd_plan_attention(*args)
        assert exc.value.status == simsd.SIMSD_ERR_INVALID_ARG
    unsupported = [(simsd.SIMSD_BF16, 4, 32, 24, 8, 128, 10, 64, 152),  # 3 heads a KV head, 192 rows
                   (simsd.SIMSD_BF16, 4, 4, 32, 8, 64, 10, 64, 152),    # bf16 needs d 128
                   (simsd.SIMSD_F32, 4, 4, 32, 8, 96, 10, 64, 152)]     # fp32 needs d 64 or 128
    for args in unsupported:
        with pytest.raises(simsd.SimsdError) as exc:
            simsd.simsd_plan_attention(*args)
        assert exc.value.status == simsd.SIMSD_ERR_UNSUPPORTED


@pytest.mark.parametrize("sms", SMS)
def test_accept_plans_match_the_rules(simsd, sms):
    for Bt, gamma, vocab in itertools.product((1, 2, 4, 8, 9, 10, 16, 64), (1, 2, 4, 8, 16, 32),
                                              (1024, 32000, 151935, 151936, 262144)):
        parts, ws = simsd.simsd_plan_accept(False, Bt, gamma, vocab, sms)
        assert (parts, ws) == (_plan.accept_parts(Bt, gamma, vocab, sms), _plan.accept_ws(Bt, gamma, vocab, sms))
        parts, ws = simsd.simsd_plan_accept(True, Bt, gamma, vocab, sms)
        assert (parts, ws) == (_plan.samp_parts(Bt, gamma, vocab, sms), _plan.samp_ws(Bt, gamma, vocab, sms))


def test_accept_decisions(simsd):
    V = 151936
    # greedy: from 4 MiB a sequence (8 x 9 rows split, the SDAR-1.7B 8 x 5 rows not)
    assert simsd.simsd_plan_accept(False, 8, 8, V, 152)[0] > 16
    assert simsd.simsd_plan_accept(False, 8, 4, V, 152) == (0, 0)
    assert simsd.simsd_plan_accept(False, 10, 16, V, 152) == (0, 0)     # more sequences than SMs / 16
    # stochastic: from 3 MiB a sequence
    assert simsd.simsd_plan_accept(True, 8, 4, V, 152)[0] > 16
    assert simsd.simsd_plan_accept(True, 1, 1, V, 152) == (0, 0)
    # one wave of at most two CTAs per SM, whatever the batch
    for sampled in (False, True):
        for Bt in range(1, 10):
            parts, _ = simsd.simsd_plan_accept(sampled, Bt, 32, V, 152)
            assert parts == 0 or Bt * parts <= 2 * 152
    with pytest.raises(simsd.SimsdError):
        simsd.simsd_plan_accept(True, 1, 33, V, 152)
    with pytest.raises(simsd.SimsdError):
        simsd.simsd_plan_accept(False, 1, 4, V, 0)
    assert simsd.simsd_plan_accept(False, 0, 4, V, 152) == (0, 0)
