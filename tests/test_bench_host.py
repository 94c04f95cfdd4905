"""Host logic of the bench: the sweep span of two overlapping launches and the source hash that
keys the recorded DRAM traffic (no GPU)."""
import bench


class FakeEvent:
    def __init__(self, t_ms):
        self.t = t_ms

    def elapsed_time(self, other):
        return other.t - self.t


def _span(q0, q1, p0, p1):
    return bench.sweep_span_ms(FakeEvent(q0), FakeEvent(q1), FakeEvent(p0), FakeEvent(p1))


def test_span_serial_launches():
    assert _span(0.0, 0.2, 0.2, 0.4) == 0.4


def test_span_overlapping_launches():
    # verifier rows start with the proposal rows and end last
    assert abs(_span(0.0, 0.27, 0.001, 0.372) - 0.372) < 1e-12
    # the verifier launch ends first
    assert abs(_span(0.0, 0.3, 0.05, 0.25) - 0.3) < 1e-12


def test_span_when_verifier_starts_first():
    assert abs(_span(0.1, 0.3, 0.0, 0.2) - 0.3) < 1e-12


def test_sweep_hash_ignores_comments_and_blank_lines(tmp_path, monkeypatch):
    src = tmp_path / "k.cu"
    src.write_text("int f() {\n  return 1;  // one\n}\n")
    monkeypatch.setattr(bench, "SWEEP_KERNEL_SRC", str(src))
    h0 = bench.sweep_source_hash()
    src.write_text("// header comment\nint f() {\n\n  return 1;   // another comment\n}\n")
    assert bench.sweep_source_hash() == h0
    src.write_text("int f() {\n  return 2;\n}\n")
    assert bench.sweep_source_hash() != h0
