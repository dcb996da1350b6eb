"""The bench's printed line (CPU only, no GPU): compact() keeps the contract's
keys in full, reduces every extra to scalars and short strings (so a parser
that keeps scalar fields one level deep sees them), and both arms report the
same `config`."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _result():
    rl = {"bound": "hbm", "kernel": "dense_tcgen05", "achieved": 6700.0, "peak": 6780.4,
          "unit": "GB/s", "frac": 0.988, "traffic": 5540048256, "bytes_per_launch": 5346660352,
          "avg_launch_us": 798.0, "bracketed_avg_us": 850.0}
    return {
        "metric": bench.METRIC, "value": 6700.0, "unit": "GB/s", "n_gpus": 1, "steps": 20,
        "warmup": 5, "ms_per_step": 20.7, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": bench.headline_config(26, 1), "roofline": rl,
        "e2e": {"value": 6000.0, "unit": "GB/s", "h2d_bytes_per_step": 1, "d2h_bytes_per_step": 1},
        "gpu_launches": 1040, "clocks": {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []},
        "cpu_baseline": {"value": 0.08, "unit": "GB/s", "cores": 16, "kind": "oracle", "sample": "x"},
        "decode_8b": {"value": 5300.0, "steps": 2000, "ms_per_step": 0.044, "roofline": dict(rl),
                      "steps20_ms_per_step": 0.046, "tokens_per_s": 1.4e6, "e2e": {"value": 4400.0},
                      "device_status": 0},
        "prefill": {"tflops": 1246.0, "ms": 23.1, "tokens_per_s": 1.4e7, "device_status": 0,
                    "roofline": dict(rl, achieved=1292.0, frac=0.68, peak=1895.9)},
        "mixed": {"ms_per_step": 0.84, "decode_tokens_per_s": 3e5, "device_status": 0,
                  "kernels_per_step": {"prefill_pair_tcgen05": {"tflops": 1190.0},
                                       "dense_tcgen05": {"gbs": 5800.0}}},
        "movement": {"reload": {"B_gbs": 197.0}, "offload": {"B_gbs": 181.0},
                     "reload_direct": {"B_gbs": 208.0}, "offload_direct": {"B_gbs": 192.0},
                     "h2d_copy": {"B_gbs": 210.0}, "mu_over_B_swap_ns_per_token": {"reload": 20.8},
                     "rows": [{"round_trip_bit_exact": True}]},
        "redo": {"rows": [{"tokens": 256, "decode_redo_kernel_ms": 5.3, "prefill_rebuild_kernel_ms": 0.08,
                           "T_decode_us_per_token": 21.0}], "device_status": 0},
        "coresidency": {"budget_tokens": 49152, "suffix_tokens": 2048,
                        "series": {"16384": [{"resident_prefixes": k, "batch": b, "step_us": 44.0,
                                              "tokens_per_s": 3e5} for k, b in ((1, 16), (2, 8))],
                                   "4096": [{"resident_prefixes": k, "batch": b, "step_us": 43.0,
                                             "tokens_per_s": 4e5} for k, b in
                                            ((1, 22), (2, 20), (3, 18), (4, 16), (6, 12), (8, 8))]},
                        "grouped_over_alternating_tokens_per_s": 2.17},
        "sched": {"tasks": 40, "decisions": 116, "native_decide_us_mean": 24.0,
                  "native_decide_us_max": 85.0, "preemptions": 16, "prefix_moves_in": 11,
                  "mean_jct_s": 11.4, "device_status": 0, "cpu_baseline": {"value": 6600.0}},
    }


def test_compact_line_keeps_contract_keys_and_flattens_extras():
    res = _result()
    line = bench.compact(res)
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "roofline",
              "e2e", "gpu_launches", "clocks", "cpu_baseline"):
        assert line[k] == res[k], k
    for extra in ("decode_8b", "prefill", "mixed", "movement", "redo", "coresidency", "sched"):
        assert extra in line, extra
        for k, v in line[extra].items():
            assert isinstance(v, (int, float, str, bool)) or v is None, (extra, k)
            if isinstance(v, str):
                assert len(v) < 120, (extra, k)
    assert line["coresidency"]["p4096_batch"] == "22,20,18,16,12,8"
    assert line["prefill"]["frac"] == 0.68
    assert len(json.dumps(line)) < 6000


def test_both_arms_report_the_same_config(monkeypatch):
    ours = bench.headline_config(bench.LAYERS_70B, 1)
    assert ours["bytes_per_step"] == ours["bytes_per_layer"] * bench.LAYERS_70B
    assert len(ours["workload"]) < 120

    class Args:
        steps, warmup, layers_70b = 2, 3, bench.LAYERS_70B

    # the oracle timing itself is replaced by a stub: only the line's fields are checked
    monkeypatch.setattr(bench, "cpu_baseline", lambda **kw: {
        "value": 0.1, "unit": "GB/s", "cores": 1, "kind": "oracle", "sample": "stub", "seconds": 2.0})
    ref = bench.run_reference(Args, 0, 1)
    assert ref["impl"] == "reference"
    assert ref["config"] == ours
    assert ref["metric"] == bench.METRIC and ref["unit"] == "GB/s" and ref["higher_is_better"]
    assert ref["steps"] == 2 and ref["warmup"] == 3
    assert ref["e2e"]["h2d_bytes_per_step"] == 0 and ref["e2e"]["value"] == ref["value"]
    assert bench.run_reference(Args, 1, 2) is None   # other ranks print nothing
