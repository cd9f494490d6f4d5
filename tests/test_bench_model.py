"""Host-side accounting of the benchmark: which path and how many launches a
workload takes, and the byte models the roofline fractions divide by."""
import bench
from paper_2609_06663_gb300.workloads import CONFIGS, sweep_workload


def test_paths_and_launch_counts():
    # bf16 heads of at least 128 keys take the tensor-core kernel, one launch
    # per group of at most 120 window rows, then the finalize and the gather
    assert bench.tensor_path(CONFIGS["c3_b10"]) and bench.row_groups(CONFIGS["c3_b10"]) == 1
    assert bench.launches_per_call(CONFIGS["c3_b10"]) == 3
    # g W = 4 * 32 = 128 window rows: two groups
    w32 = sweep_workload(4096, 32)
    assert bench.row_groups(w32) == 2 and bench.launches_per_call(w32) == 4
    assert bench.row_groups(sweep_workload(4096, 16)) == 1
    # fp32 takes the two CUDA-core passes
    assert not bench.tensor_path(CONFIGS["c0"]) and bench.launches_per_call(CONFIGS["c0"]) == 4


def test_byte_models_of_the_32k_workload():
    w = CONFIGS["c3_b10"]
    m = bench.byte_model(w)
    # K: 28 layers x 4 heads x 32768 keys x 128 dims x 2 bytes
    assert m["k"] == 28 * 4 * 32768 * 128 * 2 == 939_524_096
    # window queries: 28 layers x 28 query heads x 8 rows x 128 x 2
    assert m["q"] == 28 * 28 * 8 * 128 * 2
    kept = 28 * 4 * 3277 * 128 * 2
    assert m["kept_rows"] == kept
    # ALG: K and the queries once, the kept V rows read, kept K and V written, the indices
    assert m["alg"] == m["k"] + m["q"] + 3 * kept + 28 * 4 * 3277 * 4
    # BL counts a full read of V the pass never performs
    assert m["bl"] == 2 * m["k"] + m["q"] + 2 * kept
    assert m["alg"] < m["bl"]
