"""Host-side helpers of bench.py: algorithmic byte counts, the profile rows' source-hash
provenance (a row captured on another version of its kernel reads as null), and the
max-over-ranks aggregation rule."""
import os

import pytest

import bench


def test_gla_bytes_per_token_head_and_state():
    # q, k, v bf16 + log-gates f32 + o f32 = 14 B per (token, dim) and head; the state read and
    # written once per head; 64 KiB per emitted checkpoint at d = 128
    assert bench.gla_bytes(1, 1, 128, 1, 0) == 128 * 14 + 2 * 128 * 128 * 4
    assert bench.gla_bytes(9, 16, 128, 256, 1) == 9 * 16 * (256 * 1792 + 3 * 65536)


def test_kv_bytes_read_plus_write():
    assert bench.kv_bytes(48, 256, 65536) == 2 * 48 * 256 * 65536


def test_source_hash_ignores_comments():
    assert bench._strip_comments("a /* x\n y */ b // z\nc") == "a b c"
    assert bench._strip_comments("a\n// one\n// two\nb") == bench._strip_comments("a // one\nb")


def test_source_hash_names_the_kernel_source():
    h = bench.source_hash("gla_decode_kernel<128>")
    assert len(h) == 12 and h == bench.source_hash("gla_decode_kernel@anything")
    assert h != bench.source_hash("slot_copy_kernel")


def test_source_files_follow_the_include_graph():
    base = lambda k: [os.path.basename(f) for f in bench.source_files(k)]
    tc, dec = base("gla_chunked_tc_kernel"), base("gla_decode_kernel<128>")
    assert tc[0] == "gla_chunked_tc.cu" and dec[0] == "gla_decode.cu"
    for h in ("gla_chunk_common.cuh", "sm100_ptx.cuh", "hs_internal.cuh", "hs.h"):
        assert h in tc
    # the decode kernel's hash does not move when only the prefill's headers change
    assert "gla_chunk_common.cuh" not in dec and "sm100_ptx.cuh" not in dec
    assert "hs_internal.cuh" in dec and "hs.h" in dec
    assert base("kv_gather_kernel") == base("kv_scatter_kernel")


def test_stale_profile_rows_read_as_null(tmp_path, monkeypatch):
    fresh = bench.source_hash("gla_decode_kernel")
    (tmp_path / "dram_traffic.txt").write_text(
        "# kernel bytes hash capture\n"
        f"gla_decode_kernel<128> 1234 {fresh} x.md shape words\n"
        "slot_copy_kernel@long24 999 000000000000 y.md\n")
    (tmp_path / "tensor_pipe.txt").write_text(
        f"gla_decode_kernel@a 0.5 0.25 {fresh} z.md\n"
        "gla_chunked_tc_kernel 0.1 0.05 ffffffffffff w.md\n")
    monkeypatch.setattr(bench, "PROFILES", str(tmp_path))
    t = bench._traffic()
    assert t["gla_decode_kernel<128>"] == 1234
    assert t["slot_copy_kernel@long24"] is None
    tp = bench._tensor_pipe()
    assert tp["gla_decode_kernel@a"]["active"] == 0.5 and tp["gla_decode_kernel@a"]["source"] == "ncu z.md"
    assert tp["gla_chunked_tc_kernel"] is None


def test_committed_profile_rows_parse():
    # every committed row names a known kernel and carries a 12-digit hash
    for name, ncols in (("dram_traffic.txt", 1), ("tensor_pipe.txt", 2)):
        rows = bench._profile_rows(name, ncols)
        assert rows, name
        for kern in rows:
            assert kern.split("@")[0].split("<")[0] in bench.KERNEL_SRC


def test_aggregate_value_is_whole_job():
    assert bench.aggregate_value(2880, 30, 2, 0.1) == pytest.approx(2880 * 30 * 2 / 0.1)
    assert bench.max_over_ranks(3.5, 1) == 3.5
