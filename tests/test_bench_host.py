"""Host-side logic of bench.py that needs no GPU: the per-unit DRAM traffic
table written from an ncu CSV, and when the bench may use it."""

import csv
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _fake_csv(path, rows):
    with open(path, "w", newline="") as f:
        f.write("==PROF== a profiler banner line that the parser must skip\n")
        w = csv.writer(f, quoting=csv.QUOTE_ALL)
        w.writerow(["ID", "Kernel Name", "Metric Name", "Metric Unit", "Metric Value"])
        for i, (kernel, metric, unit, value) in enumerate(rows):
            w.writerow([i, kernel, metric, unit, value])


def test_write_traffic_averages_launches_and_scales_units(tmp_path):
    src = tmp_path / "t.csv"
    fused = "void k2_fused_l2<bf16_t, bf16_t, 512, 4, 0, 0>(FusedArgs)"
    _fake_csv(src, [
        (fused, "dram__bytes_read.sum", "Gbyte", "2.0"),
        (fused, "dram__bytes_write.sum", "Mbyte", "1,000"),
        (fused, "dram__bytes_read.sum", "Gbyte", "4.0"),
        (fused, "dram__bytes_write.sum", "Mbyte", "3,000"),
        (fused, "gpu__time_duration.sum", "us", "500"),
        ("void k1_logprob_vec<bf16_t, 256, 8, 0>(x)", "dram__bytes_read.sum", "byte", "4096"),
        ("void k1_logprob_vec<bf16_t, 256, 8, 0>(x)", "dram__bytes_write.sum", "byte", "40"),
        ("void k3_ewma_vec<256, 4>(x)", "dram__bytes_read.sum", "Gbyte", "8"),
        ("void k3_ewma_vec<256, 4>(x)", "dram__bytes_write.sum", "Gbyte", "4"),
        ("void k0_count_valid<1024>(x)", "dram__bytes_read.sum", "byte", "99"),
    ])
    out_path = tmp_path / "traffic.json"
    out = bench.write_traffic(str(src), "agentic_bf16_v151936", 151936, T=10, n_valid=5,
                              n_params=1_000_000_000, command="cmd", path=str(out_path))
    k = out["kernels"]
    assert set(k) == {"k12_decoupled_loss_fused", "k1_token_logprob", "k3_ewma_update"}
    f = k["k12_decoupled_loss_fused"]
    assert f["launches"] == 2
    assert abs(f["read_per_valid_token"] - 3.0e9 / 5) < 1e-3      # mean of 2 and 4 GB, per valid token
    assert abs(f["write_per_token"] - 2.0e9 / 10) < 1e-3          # mean of 1 and 3 GB, per token
    assert k["k1_token_logprob"]["read_per_token"] == 409.6
    assert k["k3_ewma_update"]["read_per_param"] == 8.0 and k["k3_ewma_update"]["write_per_param"] == 4.0
    assert f["source_hash"] == bench.kernel_source_hash("k12_decoupled_loss_fused")


def test_traffic_is_used_only_for_the_captured_batch(tmp_path):
    src = tmp_path / "t.csv"
    _fake_csv(src, [("void k2_loss_l2<bf16_t, bf16_t, 512, 8, 0>(K2Args)", m, "byte", "1000")
                    for m in ("dram__bytes_read.sum", "dram__bytes_write.sum")]
              + [("void k3_ewma_vec<256, 4>(x)", m, "byte", "1000")
                 for m in ("dram__bytes_read.sum", "dram__bytes_write.sum")])
    path = str(tmp_path / "traffic.json")
    bench.write_traffic(str(src), "agentic_bf16_v151936", 151936, 10, 5, 100, "cmd", path=path)
    same = bench.ncu_traffic("agentic_bf16_v151936", 151936, path=path)
    assert set(same) == {"k2_decoupled_loss_fwd_bwd", "k3_ewma_update"}
    # another batch: per-token bytes do not carry over, per-parameter bytes do
    assert set(bench.ncu_traffic("grpo_bf16_v32000", 32000, path=path)) == {"k3_ewma_update"}
    assert set(bench.ncu_traffic("agentic_bf16_v151936", 50000, path=path)) == {"k3_ewma_update"}
    tr = bench.ncu_traffic("agentic_bf16_v151936", 151936, path=path)
    assert bench.traffic_bytes(tr, "k2_decoupled_loss_fwd_bwd", T=20, n_valid=10, n_params=0) == \
        round(10 * 200 + 20 * 100)
    assert bench.traffic_bytes(tr, "k1_token_logprob", T=20, n_valid=10, n_params=0) is None


def test_partial_capture_keeps_unchanged_kernels_and_drops_stale_ones(tmp_path):
    # a capture of one kernel rewrites its entry and keeps the others while their
    # sources hash as recorded; an entry whose hash no longer matches is dropped
    import json
    path = str(tmp_path / "traffic.json")
    both = tmp_path / "both.csv"
    _fake_csv(both, [("void k2_loss_l2<bf16_t, bf16_t, 512, 8, 0>(K2Args)", m, "byte", "1000")
                     for m in ("dram__bytes_read.sum", "dram__bytes_write.sum")]
              + [("void k3_ewma_vec<256, 4>(x)", m, "byte", "1000")
                 for m in ("dram__bytes_read.sum", "dram__bytes_write.sum")])
    bench.write_traffic(str(both), "agentic_bf16_v151936", 151936, 10, 5, 100, "cmd", path=path)
    one = tmp_path / "one.csv"
    _fake_csv(one, [("void k3_ewma_vec<256, 4>(x)", m, "byte", "3000")
                    for m in ("dram__bytes_read.sum", "dram__bytes_write.sum")])
    out = bench.write_traffic(str(one), "agentic_bf16_v151936", 151936, 10, 5, 100, "cmd", path=path)
    assert set(out["kernels"]) == {"k2_decoupled_loss_fwd_bwd", "k3_ewma_update"}
    assert out["kernels"]["k3_ewma_update"]["read_per_param"] == 30.0
    assert out["kernels"]["k2_decoupled_loss_fwd_bwd"]["read_per_valid_token"] == 200.0
    d = json.load(open(path))
    d["kernels"]["k2_decoupled_loss_fwd_bwd"]["source_hash"] = "stale"
    json.dump(d, open(path, "w"))
    out = bench.write_traffic(str(one), "agentic_bf16_v151936", 151936, 10, 5, 100, "cmd", path=path)
    assert set(out["kernels"]) == {"k3_ewma_update"}
    # a capture of another batch starts a new table
    out = bench.write_traffic(str(one), "grpo_bf16_v32000", 32000, 10, 5, 100, "cmd", path=path)
    assert set(out["kernels"]) == {"k3_ewma_update"} and out["workload"] == "grpo_bf16_v32000"


def test_shared_workload_config_keys():
    class A:
        workload, ewma_n, tau = "agentic_bf16_v151936", 100, 0.5

    class B:
        T, V, rd_lo, rd_hi, eps_low, eps_high = 8, 16, 0.5, 2.0, 0.2, 0.28

        class z_theta:
            dtype = "torch.bfloat16"

            @staticmethod
            def element_size():
                return 2

    cfg = bench.workload_config(A, B, 6, 1)
    assert cfg["T"] == 8 and cfg["V"] == 16 and "6 valid" in cfg["workload"]
    assert cfg["parallelism"] == "single GPU"
    assert bench.workload_config(A, B, 6, 4)["parallelism"] == "replicas x4"


def test_reference_arm_runs_the_oracle_alone(tmp_path):
    """The oracle arm: no build and no CUDA library in its process, ms_per_step
    is the time its sample steps took, and value is the tokens they processed
    per second (nothing extrapolated)."""
    import json
    import subprocess
    import time
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
           "--workload", "tiny_f32_v4096", "--steps", "3", "--warmup", "1",
           "--ewma-n", "1000000"]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    t0 = time.time()
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=300, env=env, cwd=tmp_path)
    wall = time.time() - t0
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["repo_libs_loaded"] == []
    S = line["config"]["sample_tokens_per_step"]
    assert S == 256 and line["config"]["sample_ewma_params_per_step"] == 1000000
    assert abs(line["value"] - S / (line["ms_per_step"] / 1e3)) <= 1e-3 * line["value"]
    assert line["steps"] * line["ms_per_step"] / 1e3 < wall
    assert line["e2e"]["value"] == line["value"] == line["cpu_baseline"]["value"]
