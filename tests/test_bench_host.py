"""Host-side helpers of bench.py that need no GPU: the comment-blind source
digest that keys the committed DRAM-traffic record, the rule that the record
is reported only while the kernel sources match it, and the workload config
shared by the CUDA arm and the oracle arm."""

import contextlib
import io
import json
import types

import bench
from paper_2603_18599_gb300 import workloads


def test_comment_removal_keeps_code_and_string_literals():
    src = ('int a = 1; // trailing\n'
           '\n'
           '/* block\n   comment */ int b = 2;\n'
           'const char* s = "// not a comment";\n'
           "char c = '/';  /* x */\n")
    out = bench.code_without_comments(src)
    assert out.split("\n") == ['int a = 1;', ' int b = 2;', 'const char* s = "// not a comment";',
                               "char c = '/';"]


def test_digest_ignores_comments_but_not_code(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2603_18599_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))

    def digest(body):
        for f in bench.KERNEL_SOURCES:
            (csrc / f).write_text(body)
        return bench.kernel_source_digest()

    base = digest("int x = 1;\n")
    assert digest("// a comment\nint x = 1;  /* another */\n\n") == base
    assert digest("int x = 2;\n") != base


def _record(path, sha, nbytes):
    path.write_text("# a capture\nsource_sha256: %s\ndram_bytes_read: 1\ndram_bytes_write: 2\n"
                    "dram_bytes_per_launch: %d\n" % (sha, nbytes))


def test_traffic_reported_only_while_the_sources_match(tmp_path, monkeypatch):
    rec = tmp_path / "traffic.txt"
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(rec))
    _record(rec, bench.kernel_source_digest(), 12345)
    assert bench.measured_traffic() == 12345
    _record(rec, "0" * 64, 12345)
    assert bench.measured_traffic() is None
    rec.unlink()
    assert bench.measured_traffic() is None


def test_committed_traffic_record_parses():
    """The committed record has every field; its byte count is the sum of
    its read and write counters."""
    rec = {}
    with open(bench.TRAFFIC_FILE) as fh:
        for ln in fh:
            if ln.startswith("#") or ":" not in ln:
                continue
            k, v = ln.split(":", 1)
            rec[k.strip()] = v.strip()
    assert len(rec["source_sha256"]) == 64
    assert int(rec["dram_bytes_per_launch"]) == int(rec["dram_bytes_read"]) + int(rec["dram_bytes_write"])


def test_reference_arm_line_uses_the_shared_workload_config(monkeypatch):
    monkeypatch.setattr(bench, "dist_env", lambda: (0, 0, 1))
    args = types.SimpleNamespace(steps=1, warmup=0, gpus=1)
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.run_reference(args)
    line = json.loads(buf.getvalue().strip().splitlines()[-1])
    wl = workloads.workloads()[bench.WORKLOAD]
    assert line["impl"] == "reference"
    assert line["config"] == bench.workload_config(wl)
    assert line["metric"] == bench.METRIC and line["unit"] == "positions/s" and line["higher_is_better"]
    assert line["e2e"]["value"] == line["value"] and line["cpu_baseline"]["value"] == line["value"]
    assert line["value"] > 0
