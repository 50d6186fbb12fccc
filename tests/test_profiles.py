"""Consistency of the committed ncu summaries (profiles/) with the sources they describe:
the Gram DRAM-traffic figure that bench.py reports is only valid for the Gram kernel source
it was measured on, and every summary is short text whose commands run committed files."""
import importlib.util
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROFILES = os.path.join(ROOT, "profiles")


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_gram_traffic_summary_matches_kernel_source():
    """The summary's source_sha256 is the current Gram kernel's (else bench.py reports
    traffic null): change the kernel, then re-capture its DRAM counters."""
    b = _bench()
    traffic = b.profiled_traffic("llama7b_attn_4096")
    assert traffic is not None
    # the algorithmic minimum is the two bf16 operands (2 x 2.15 GB); more is re-reads
    assert 4.0e9 < traffic < 1.0e10


def test_profiles_are_short_text_with_committed_commands():
    names = sorted(os.listdir(PROFILES))
    assert names, "no profile summaries"
    for name in names:
        path = os.path.join(PROFILES, name)
        assert name.endswith((".md", ".txt")), name
        assert os.path.getsize(path) < 16384, name
        text = open(path).read()
        # commands name only committed files (no scratch paths or tool wrappers)
        assert "_work" not in text and "gpurun" not in text, name
        assert "ncu " in text, f"{name} gives no ncu command"
        assert "--clock-control none" in text, name
