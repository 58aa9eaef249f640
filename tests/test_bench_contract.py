"""The benchmark's reference arm (the CPU oracle) runs without a GPU and prints one JSON line
with the keys the benchmark contract names, on the same metric and workload as the GPU arm."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "1"], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["config"]["workload"] == "n32768_kl256_ku256"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["e2e"]["value"] == d["value"]


def test_trace_summary_of_a_synthetic_timeline():
    """The timeline summary of `bench.py --trace` on a constructed record whose intervals are
    known: a 100-unit panel period with fixed offsets for every stamp."""
    import numpy as np

    sys.path.insert(0, ROOT)
    import bench

    cap, npan = 64, 40
    T = np.zeros((4, cap, 16), dtype=np.int64)
    q = np.arange(npan)
    A = T[0]
    A[q, 0] = 1000 + 100 * q          # panel start
    for k in range(4):                # column steps: start, barrier, records sent
        A[q, 4 + 3 * k] = A[q, 0] + 5 + 20 * k
        A[q, 5 + 3 * k] = A[q, 4 + 3 * k] + 7
        A[q, 6 + 3 * k] = A[q, 5 + 3 * k] + 9
    A[q, 1] = A[q, 6 + 3 * 2]         # step 2's records sent
    A[q, 2] = A[q, 1] + 30            # panel done
    A[q, 3] = A[q, 2] + 4             # next block usable
    S1 = T[1]
    S1[q, 0] = A[q, 0] - 50
    S1[q, 1] = S1[q, 0] + 11
    S1[q, 2] = A[q, 1] + 2
    S1[q, 3] = A[q, 1] + 6
    S1[q, 4] = S1[q, 3] + 13
    S2 = T[2]
    S2[q, 0] = A[q, 0] - 300
    S2[q, 1] = S2[q, 0] + 17
    S2[q, 3] = A[q, 2] + 19
    S2[q, 4] = (1000 + 100 * (q + 1) - 50) - 23   # streamer 1 has block q+2 (its entry q+1) 23 later
    L = T[3]
    L[q, 0] = A[q, 0] - 500
    L[q, 1] = L[q, 0] + 40
    out = bench.trace_summary(T, 8, 32)
    a = out["panel_cta"]
    assert a["period"]["median"] == 100 and a["period"]["p90"] == 100
    assert a["wait_for_next_block"]["mean"] == 4
    assert a["step2_records_sent_to_panel_done"]["median"] == 30
    assert a["block_in_to_next_panel_start"]["median"] == A[11, 0] - A[10, 3]
    for k in range(4):
        assert a[f"step{k}_start_to_barrier"]["median"] == 7
        assert a[f"step{k}_barrier_to_records_sent"]["median"] == 9
    assert a["panel_start_to_step0_start"]["median"] == 5
    s1 = out["streamer1"]
    assert s1["block_in_to_first_records"]["median"] == 11
    assert s1["last_records_wait_starts_after_sent"]["median"] == 2
    assert s1["last_records_seen_after_sent"]["median"] == 6
    assert s1["last_step_and_band_send"]["median"] == 13
    assert s1["band_sent_to_panel_cta_has_block"]["median"] == A[10, 3] - S1[10, 4]
    s2 = out["streamer2"]
    assert s2["block_in_to_first_records"]["median"] == 17
    assert s2["last_records_seen_after_panel_cta_done"]["median"] == 19
    assert s2["band_sent_to_streamer1_block_in"]["median"] == 23
    assert out["loader_wait_for_hand_over"]["median"] == 40
    assert out["panel_done_to_hand_over_seen"]["median"] == L[20, 1] - A[15, 2]
