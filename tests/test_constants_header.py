"""The kernels' constants header is exactly what its generator writes (exact
integer arithmetic; no drift between the committed header and the script),
and the generator's own checks (one threshold per rank-table bucket, a rank
step of exactly 1 there) hold while it runs."""
import importlib.util
import io
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_10010_gb300", "csrc")


def test_header_matches_generator():
    spec = importlib.util.spec_from_file_location("gen_constants", os.path.join(CSRC, "gen_constants.py"))
    gen = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(gen)
    buf = io.StringIO()
    gen.main(buf)
    with open(os.path.join(CSRC, "curvefp_constants.h")) as f:
        assert buf.getvalue() == f.read()
