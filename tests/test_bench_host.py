"""Host-side logic of bench.py: workload shapes, steady-state starts, rank reduction (gloo, 2 ranks),
and the reference (oracle) arm's JSON line."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def test_workloads_match_the_stated_configs():
    w = bench.WORKLOADS
    assert (w[1]["L"], w[1]["H"], w[1]["KVH"], w[1]["B"], w[1]["lp"], w[1]["K"], w[1]["r"]) == (1, 32, 8, 1, [128], 256, 64)
    assert (w[2]["L"], w[2]["H"], w[2]["KVH"], w[2]["B"], w[2]["lp"][0], w[2]["K"]) == (36, 32, 8, 16, 512, 2048)
    assert w[2]["key_scale"]
    assert (w[3]["L"], w[3]["H"], w[3]["KVH"], w[3]["B"], w[3]["lp"][0], w[3]["K"]) == (40, 40, 8, 64, 2048, 4096)
    assert (w[4]["L"], w[4]["H"], w[4]["KVH"], w[4]["B"], w[4]["lp"][0], w[4]["K"]) == (64, 64, 8, 32, 1024, 8192)
    assert (w[5]["L"], w[5]["H"], w[5]["KVH"], w[5]["B"], w[5]["K"]) == (40, 40, 10, 48, 4096)
    assert min(w[5]["lp"]) >= 256 and max(w[5]["lp"]) <= 4096 and len(set(w[5]["lp"])) > 10
    assert min(w[5]["gen"]) >= 8192 and max(w[5]["gen"]) <= 32768
    assert all(x["r"] == 64 for x in w.values())


@pytest.mark.parametrize("cfg", [2, 3, 4, 5])
def test_steady_state_is_a_reachable_state(cfg):
    w = bench.WORKLOADS[cfg]
    g0, c0 = bench.steady_state(w)
    for g, c, gen in zip(g0, c0, w["gen"]):
        phase = g % w["r"]
        assert c == w["K"] + w["r"] + phase  # c right after an eviction, plus the appends since
        assert g - phase >= w["K"] + 2 * w["r"]  # that eviction step is one the trigger can reach
        assert g + 2048 <= gen  # the sequence stays active through a benchmark window


@pytest.mark.parametrize("cfg", [2, 3, 4])
def test_equal_length_batches_spread_their_evictions_over_every_window(cfg):
    """Sequence b of an equal-length batch evicts on the steps where its generated count reaches a
    multiple of r; with the phases spread over [0, r), any window of W steps holds about W B / r
    (sequence) rounds, so a short timed window still prices the eviction."""
    w = bench.WORKLOADS[cfg]
    g0, _ = bench.steady_state(w)
    r, B = w["r"], w["B"]
    fires = [sum(1 for g in g0 if (g + t + 1) % r == 0) for t in range(3 * r)]
    for W in (20, 32, r):
        for t0 in range(2 * r):
            n = sum(fires[t0:t0 + W])
            assert abs(n - W * B / r) <= 1 + (B // r), (W, t0, n)
    assert sum(fires[:r]) == B  # every sequence once per r steps


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_main(rank, world, port, q):
    import torch.distributed as dist

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms, units = bench.reduce_over_ranks(10.0 + rank, 16.0, world)
    q.put((rank, ms, units))
    dist.destroy_process_group()


def test_reduce_over_ranks_gloo_two_ranks():
    import torch.multiprocessing as mp

    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    # time = max over ranks, units = sum over ranks (weak scaling: every rank runs its own batch)
    assert got == [(0, 11.0, 32.0), (1, 11.0, 32.0)]


def test_reference_arm_prints_one_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "1",
                          "--steps", "1", "--warmup", "3", "--cpu-seconds", "0.4"],
                         capture_output=True, text=True, timeout=300, check=True).stdout
    lines = [l for l in out.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
    assert d["metric"] == bench.METRIC


def _attn_totals(us, by):
    return {"us_per_launch": us, "bytes_per_launch": by, "algorithmic_GBps": by / (us * 1e-6) / 1e9}


def test_roofline_takes_the_windowed_duration_of_the_eviction_free_steps():
    peaks = {"hbm_gbs": 6000.0}
    a = _attn_totals(40.0, 180e6)  # serialized: per-launch events
    # two eviction-free steps of 36 launches each: 1.26 ms and 1.26 ms, 36 x 174 MB each
    clean = [(1.26, 36, 36 * 174e6), (1.26, 36, 36 * 174e6)]
    r = bench.attention_roofline(a, clean, 4, 36, peaks, "measured", 178e6)
    assert r["us_per_launch"] == pytest.approx(1000.0 * 2.52 / 72)
    assert r["algorithmic_bytes_per_launch"] == pytest.approx(174e6)
    assert r["achieved"] == pytest.approx(174e6 / (35e-6) / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / 6000.0)
    assert r["frac_of_nominal_8TBps"] == pytest.approx(r["achieved"] / 8000.0)
    assert r["serialized"]["us_per_launch"] == 40.0
    assert r["serialized"]["frac"] == pytest.approx(180e6 / 40e-6 / 1e9 / 6000.0)
    assert r["traffic"] == 178e6 and r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert "2 of 4 steps" in r["timing"] and "36 layers" in r["timing"]


def test_roofline_falls_back_to_the_per_launch_events_without_eviction_free_steps():
    a = _attn_totals(240.0, 1.6e9)
    r = bench.attention_roofline(a, [], 128, 40, {"hbm_gbs": 6691.0}, "fallback", None)
    assert r["us_per_launch"] == 240.0 and r["algorithmic_bytes_per_launch"] == 1.6e9
    assert r["achieved"] == pytest.approx(a["algorithmic_GBps"])
    assert r["timing"] == r["serialized"]["timing"] and r["peak_source"].startswith("fallback")
    assert r["traffic"] is None
    assert bench.attention_roofline(None, [], 1, 1, {"hbm_gbs": 1.0}, "measured", None) is None


def _kern(us, by, n):
    return {"launches": n, "ms_total": us * n / 1000.0, "us_per_launch": us, "bytes_per_launch": by,
            "algorithmic_GBps": by / (us * 1e-6) / 1e9}


def test_eviction_roofline_prices_the_copy_kernel_and_the_round():
    peaks = {"hbm_gbs": 6000.0}
    kern = {"attn": _kern(200.0, 1.2e9, 640), "select": _kern(10.0, 0.0, 20), "compact": _kern(20.0, 68e6, 20)}
    r = bench.eviction_roofline(kern, 20, peaks, "measured", 70e6)
    assert r["kernel"].startswith("compact_kernel") and r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(68e6 / 20e-6 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / 6000.0)
    assert r["frac_of_nominal_8TBps"] == pytest.approx(r["achieved"] / 8000.0)
    assert r["round"]["us_per_round"] == pytest.approx(30.0)
    assert r["round"]["bytes_per_round"] == pytest.approx(68e6)
    assert r["round"]["frac"] == pytest.approx(68e6 / 30e-6 / 1e9 / 6000.0)
    assert r["traffic"] == 70e6 and r["launches"] == 20
    # the fused kernel, when present, is the one priced; order-free select reported beside it
    kern2 = {"evict": _kern(12.0, 68e6, 10)}
    hole = ({"select": _kern(5.0, 2e6, 10), "stack": _kern(14.0, 33e6, 2)}, 10)
    r2 = bench.eviction_roofline(kern2, 10, peaks, "fallback", None, hole)
    assert r2["holefill_fill"]["achieved"] == pytest.approx(33e6 / 14e-6 / 1e9)
    assert r2["holefill_fill"]["us_per_round"] == pytest.approx(2.8)
    assert r2["kernel"].startswith("evict_kernel") and r2["peak_source"].startswith("fallback")
    assert r2["round"]["us_per_round"] == pytest.approx(12.0)
    assert r2["holefill_select"]["achieved"] == pytest.approx(2e6 / 5e-6 / 1e9)
    assert r2["holefill_select"]["us_per_round"] == pytest.approx(5.0)
    # the whole-stack compaction, when present, is the one priced; the others are listed beside it
    kern3 = {"stack": _kern(600.0, 4.3e9, 1), "evict": _kern(12.0, 68e6, 10), "plan": _kern(100.0, 0.0, 2)}
    r3 = bench.eviction_roofline(kern3, 74, peaks, "measured")
    assert r3["kernel"].startswith("compact_stack_kernel") and r3["launches"] == 1
    assert r3["achieved"] == pytest.approx(4.3e9 / 600e-6 / 1e9)
    assert r3["also"]["evict"]["achieved"] == pytest.approx(68e6 / 12e-6 / 1e9)
    assert r3["round"]["us_per_round"] == pytest.approx(720.0 / 74)  # the plan is not in the round
    assert r3["plan"]["launches"] == 2 and "target" in r3
    r4 = bench.eviction_roofline(kern3, 74, peaks, "measured", compaction="holefill")
    assert r4["kernel"].startswith("fill_stack_kernel")
    # no eviction in the evented pass: nothing to report
    assert bench.eviction_roofline({"attn": kern["attn"]}, 0, peaks, "measured") is None


def test_eviction_window_is_the_step_time_beyond_the_attention_bytes():
    # eviction-free steps: 2 x (1.0 ms for 6e9 attention bytes) -> 6e9 B/ms
    clean = [(1.0, 64, 6e9), (1.0, 64, 6e9)]
    # evicting steps: attention bytes 5.94e9 (0.99 ms at that rate) plus eviction time
    evicting = [(1.99 + 0.0, 5.94e9, 64, 64 * 68e6), (1.5, 5.94e9, 64, 64 * 68e6)]
    w = bench.eviction_window(clean, evicting)
    extra = (1.99 - 0.99) + (1.5 - 0.99)
    assert w["rounds"] == 128 and w["steps"] == 2
    assert w["us_per_round"] == pytest.approx(1000.0 * extra / 128)
    assert w["bytes_per_round"] == pytest.approx(68e6)
    assert w["GBps"] == pytest.approx(128 * 68e6 / (extra * 1e-3) / 1e9)
    assert bench.eviction_window([], evicting) is None and bench.eviction_window(clean, []) is None
    r = bench.eviction_roofline({"evict": _kern(12.0, 68e6, 10)}, 10, {"hbm_gbs": 6000.0}, "measured", None, None, w)
    assert r["windowed"]["frac"] == pytest.approx(w["GBps"] / 6000.0)
    assert w["resolved"] and w["noise_us_per_round"] == 0.0


def test_eviction_window_within_the_clean_steps_noise_is_not_resolved():
    # clean steps 1.00 / 1.02 ms for 6e9 bytes: the prediction itself is uncertain by ~1%
    clean = [(1.00, 64, 6e9), (1.02, 64, 6e9)]
    rate = 2.02 / 12e9
    evicting = [(5.94e9 * rate + 0.001, 5.94e9, 64, 64 * 1e6)]  # 1 us beyond the prediction
    w = bench.eviction_window(clean, evicting)
    sd = 0.01 / 6e9  # the two rates' population spread (ms per byte)
    assert w["noise_us_per_round"] == pytest.approx(1000.0 * sd * 5.94e9 / 64)
    assert not w["resolved"] and "GBps" not in w
    assert w["us_per_round_at_most"] == pytest.approx(1000.0 * (0.001 + 2 * sd * 5.94e9) / 64)
    r = bench.eviction_roofline({"stack": _kern(14.0, 33e6, 1)}, 64, {"hbm_gbs": 6000.0}, "measured", None, None, w)
    assert r["windowed"]["frac"] is None
