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
