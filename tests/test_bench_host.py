"""Host logic of the benchmark without a GPU: the CPU baseline times the oracle on one core and then on
every host core at once (one spawned process per core), and reports the all-cores rate."""
import bench
import mikv_inputs as mi


def test_cpu_baseline_one_and_all_cores():
    r = bench.cpu_baseline(mi.WORKLOADS["tiny"], seconds=1.0)
    assert r["kind"] == "oracle" and r["unit"] == bench.UNIT
    assert r["single_core_value"] > 0 and r["value"] > 0 and r["ms_per_head_step"] > 0
    if r["cores"] > 1:  # the all-cores figure was measured, on every core the process may use
        assert "all_cores_unavailable" not in r
        assert r["cores"] == len(bench.os.sched_getaffinity(0))
    else:
        assert r["value"] == r["single_core_value"]


def test_cpu_baseline_single_core_only():
    r = bench.cpu_baseline(mi.WORKLOADS["tiny"], seconds=0.2, all_cores=False)
    assert r["cores"] == 1 and r["value"] == r["single_core_value"]


def test_source_hash_ignores_comments_only():
    """The attention-source hash that gates the profiled traffic figure follows the code, not its comments."""
    a = 'int x = 1; // one\n/* block\n comment */ const char* s = "// kept"; char c = \'/\';'
    b = 'int x = 1;\nconst char* s = "// kept";   char c = \'/\';  // other'
    assert bench._code_only(a) == bench._code_only(b) == 'int x = 1; const char* s = "// kept"; char c = \'/\';'
    assert bench._code_only("a = b;") != bench._code_only("a = c;")
