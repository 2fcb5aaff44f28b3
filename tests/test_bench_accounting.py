"""The benchmark's roofline accounting: the algorithmic bytes of the probe and fused score kernels
follow their stated per-unit definitions, and the traffic figures come from the committed ncu
summaries."""
import bench


def test_score_algorithmic_bytes_per_pair_request_and_instance():
    # per pair: the u32 hit read; with per-pair outputs also f32 TPOT, f32 TTFT and the u8 class
    # written.  Per request: L (u32) and the two f32 targets read, the i32 pick and u8 path written.
    # Per instance: b, qr, B_max (i32) and q, S, M_KV (i64) read.
    R, I = 16384, 1024
    assert bench.score_algorithmic_bytes(R, I, per_pair_outputs=True) == R * I * 13 + R * 17 + I * 36
    assert bench.score_algorithmic_bytes(R, I, per_pair_outputs=False) == R * I * 4 + R * 17 + I * 36
    assert bench.score_algorithmic_bytes(0, I, True) == I * 36


def test_probe_algorithmic_bytes_from_launch_counters():
    st = {"rows_scratch": 3, "rows_derived": 5, "lookups_scratch": 100, "lookups_derived": 20,
          "chain_reads": 110, "pairs_derived": 0}
    I = 64
    nbytes, lookups = bench.probe_algorithmic_bytes(st, I, with_tpf=True)
    assert lookups == 120
    # a 32-byte sector per lookup, 8 B per chain block read, u32 hit + f32 T_pf per pair, and the
    # base row's hits (4 B per instance) a derived row starts from
    assert nbytes == 32 * 120 + 8 * 110 + 8 * I * (3 + 5) + 4 * I * 5
    nbytes0, _ = bench.probe_algorithmic_bytes(st, I, with_tpf=False)
    assert nbytes - nbytes0 == 4 * I * (3 + 5)


def test_traffic_figures_are_read_from_the_committed_profiles():
    assert bench.profile_figure("greedy_pipe_production_window_1024x8192.md", "DRAM bytes per request") > 8 * 1024
    assert bench.profile_figure("score_block_production_window_1024x16384.md", "DRAM bytes per request") > 0
    assert bench.profile_figure("probe_search_production_window_1024x16384.md", "DRAM bytes per lookup") > 32
    assert bench.profile_figure("no_such_summary.md", "DRAM bytes per request") is None


def test_job_rate_counts_every_rank():
    assert bench.job_rate(1, 1000, 10.0) == 1000 / 0.010
    assert bench.job_rate(4, 1000, 10.0) == 4 * 1000 / 0.010
