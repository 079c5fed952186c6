"""bench.py's `config` object on CPU: both arms describe the workload the same
way, by name and shape, with the protection count of the seeded mask."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))


def test_headline_config():
    import bench
    w = bench._workload(bench.parse_args_from([]))
    c = bench.workload_config(w)
    assert c["workload"] == "qwen25vl7b"
    assert (c["layers"], c["batch"], c["q_heads"], c["kv_heads"]) == (28, 1, 28, 4)
    assert c["tokens"] == "64 text + 1296 image + 100 text"
    assert (c["base"], c["bits"], c["keys_only"]) == ("minmax", 2, False)
    assert c["protected_heads"] == 14 and c["decode_steps"] == 32
    assert "l2" in c and "launch" in c


def test_overrides_rename_the_workload():
    import bench
    args = bench.parse_args_from(["--workload", "internvl25_8b", "--salient-permille", "20",
                                  "--meta-bits", "32", "--layers", "4"])
    c = bench.workload_config(bench._workload(args))
    assert c["workload"] == "internvl25_8b_meta32_4layers_salient20"
    assert c["layers"] == 4 and c["base"] == "akvq" and c["bits"] == 4


def test_dequantize_bytes_on_the_one_layer_cache(monkeypatch):
    """The dequantize side measurement counts the cache entries a decode step
    reads plus the two BF16 outputs; driven here on CPU with the library calls
    and CUDA events stubbed out."""
    import types

    import torch

    import bench
    import paper_2609_35800_gb300 as hg
    from paper_2609_35800_gb300 import build, workloads as wl
    from paper_2609_35800_gb300.runner import config_of, shape_of
    build.build()
    w = wl.WORKLOADS["tiny"]
    mask = wl.protection_mask(w).numpy()
    sh, cf = shape_of(w), config_of(w)
    cache = hg.hg_cache_create(sh, cf, mask, 1 << 40, hg.hg_cache_layout(sh, cf, mask))
    runner = types.SimpleNamespace(w=w, cache=cache)
    _, dec_b, _ = bench.geometry_bytes(runner)

    calls = []

    class Ev:
        def record(self, stream):
            pass

        def elapsed_time(self, other):
            return 0.5

    monkeypatch.setattr(torch.cuda, "Event", lambda enable_timing=True: Ev())
    monkeypatch.setattr(torch.cuda, "synchronize", lambda: None)
    monkeypatch.setattr(hg, "hg_dequantize_kv",
                        lambda c, l, n, k, v, f, s: calls.append((l, n, k.shape)))
    r = bench.time_dequantize(runner, w, dec_b, "cpu", lambda: None, None)
    # 3 quantized heads: 64 text rows + 256 coded tokens (2 x 32 code bytes,
    # 2 x 8 metadata bytes); protected head 1: 320 BF16 rows; outputs K and V
    want = 3 * (64 * 512 + 256 * 2 * (32 + 8)) + 320 * 512 + 2 * 4 * 320 * 256
    assert r["bytes"] == want and r["appended"] == 0 and r["launches"] == 1
    assert r["ms"] == 0.5 and calls == [(0, 1, (1, 1, 4, 320, 128))] * 3


def test_cpu_baseline_fields_split_quantize_and_decode():
    """The oracle's quantize GB/s and decode tokens/s from one timed sample;
    decode tokens/s scaled to all layers when the sample holds fewer."""
    import bench
    from paper_2609_35800_gb300 import workloads as wl
    w = wl.WORKLOADS["qwen25vl7b"]
    parts = {"quant_bytes": 2e9, "quant_s": 4.0, "dec_bytes": 3e9, "dec_s": 2.0}
    f = bench.cpu_baseline_fields(w, 28, 8, parts)
    assert f["quantize_GBps"] == 0.5 and f["decode_GBps"] == 1.5
    assert f["decode_tokens_per_s"] == 1 * 8 / 2.0  # batch 1, 8 steps over all 28 layers in 2 s
    assert "all 28 layers" in f["decode_tokens_per_s_basis"]
    assert f["nproc"] == os.cpu_count() and f["cpu_model"]
    g = bench.cpu_baseline_fields(w, 7, 8, parts)  # a quarter of the layers: a quarter of the time per token
    assert g["decode_tokens_per_s"] == 1 * 8 / 2.0 * 7 / 28
    assert "extrapolated from 7 of 28" in g["decode_tokens_per_s_basis"]


def test_cpu_sample_plan_and_timed_repetitions(monkeypatch):
    """The CPU baseline samples the whole workload step on the small caches
    and one layer with two decode steps on the large ones, and repeats the
    sample until the timed oracle calls reach the floor (at least once, at most
    max_reps times), summing bytes, seconds and the quantize / decode parts."""
    import bench
    from paper_2609_35800_gb300 import workloads as wl
    assert bench.cpu_sample_plan(wl.WORKLOADS["qwen25vl7b"]) == (28, 32)
    assert bench.cpu_sample_plan(wl.WORKLOADS["qwen25vl72b"]) == (1, 2)
    calls = []

    def fake(w, n_layers, n_steps, parts=None):
        calls.append((n_layers, n_steps))
        parts.update(quant_bytes=10, quant_s=0.5, dec_bytes=30, dec_s=1.5)
        return 40, 2.0, 7

    monkeypatch.setattr(bench, "oracle_sample", fake)
    w = wl.WORKLOADS["qwen25vl7b"]
    nb, secs, threads, reps, parts = bench.timed_oracle_samples(w, 28, 32, min_seconds=5.0)
    assert (reps, nb, secs, threads) == (3, 120, 6.0, 7) and calls == [(28, 32)] * 3
    assert parts == {"quant_bytes": 30, "quant_s": 1.5, "dec_bytes": 90, "dec_s": 4.5}
    f = bench.cpu_baseline_fields(w, 28, 32 * reps, parts)
    assert f["decode_tokens_per_s"] == round(1 * 96 / 4.5, 3)  # batch 1, 3 x 32 steps in 4.5 s
    calls.clear()
    assert bench.timed_oracle_samples(w, 28, 32, min_seconds=0.0)[3] == 1   # at least once
    assert bench.timed_oracle_samples(w, 28, 32, min_seconds=1e9, max_reps=4)[3] == 4


def test_floors_on_stubbed_events(monkeypatch):
    """measure_floors times three things with the same L2 flush before each
    repetition and reports medians; driven here with stub events on CPU."""
    import types

    import torch

    import bench
    ticks = iter(range(1000))
    flushes = []

    class Ev:
        def record(self, stream):
            self.t = next(ticks)

        def elapsed_time(self, other):
            return (other.t - self.t) * 1e-3  # ms: one tick = 1 us

    monkeypatch.setattr(torch.cuda, "Event", lambda enable_timing=True: Ev())
    monkeypatch.setattr(torch.cuda, "synchronize", lambda: None)
    monkeypatch.setattr(torch.cuda, "_sleep", lambda n: None)
    f = bench.measure_floors(4096, lambda: flushes.append(1), None, "cpu", reps=3)
    assert len(flushes) == 9
    assert f["events_only_us"] == 1.0 and f["empty_kernel_us"] == 1.0 and f["read_same_bytes_us"] == 1.0
    assert f["read_bytes"] == 4096 and f["read_GBps"] > 0
