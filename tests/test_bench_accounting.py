"""The benchmark's algorithmic work, checked on the CPU against per-tensor byte
counts written out here from the layouts of the C ABI.

Compulsory traffic is every input read once and every output written once, at
the dtype the benchmark stores, plus the state once per sequence.  A wider
output dtype must raise the byte count it is divided by, never the fraction.
"""
import importlib.util
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("kdn_bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _diag_token_head(d, act, out):
    # q, k, g, omega [.., d_k] and v [.., d_v] in, r one per token-head in, o [.., d_v] out
    return 4 * d * act + d * act + act + d * out


def test_forward_bytes_per_token_head(bench):
    assert _diag_token_head(128, 2, 2) == 1538
    assert bench.fwd_bytes(1, 1, 1, 128, 128, with_state=False) == 1538
    # fp32 o: 256 more bytes per token-head, in the denominator
    assert bench.fwd_bytes(1, 1, 1, 128, 128, out_bytes=4, with_state=False) == 1794


def test_forward_bytes_of_the_1p3b_layer(bench):
    B, T, H, d = 8, 4096, 16, 128
    state = B * H * (d * d * 4 + d * 4)   # S_T and p_T, fp32, once per sequence
    want = B * T * H * 1538 + state
    assert bench.fwd_bytes(B, T, H, d, d) == want
    assert abs(want / 1e6 - 814.8) < 0.5           # 814.8 MB per forward launch
    assert 95.0 < want / 8e12 * 1e6 < 110.0        # ~102 us at the 8 TB/s spec bandwidth


def test_backward_bytes_per_token_head(bench):
    d = 128
    reads = (2 * d + d + 2 * d + 1 + d) * 2       # q, k, v, g, omega, r, dO
    writes = (2 * d + d + 2 * d + 1) * 2          # dq, dk, dv, dg, domega, dr
    assert reads + writes == 2820
    per_seq = d * d * 4 + d * 4                   # dS_0, dp_0
    assert bench.bwd_bytes(1, 1, 1, d, d) == 2820 + per_seq
    B, T, H = 8, 4096, 16
    assert abs(bench.bwd_bytes(B, T, H, d, d) / 1e6 - 1487.0) < 1.0


def test_decode_bytes_per_head_step(bench):
    d = 128
    state = 2 * (d * d * 4 + d * 4)               # S and p read and written, fp32
    ins = (4 * d + d + 1) * 2                     # q, k, g, omega, v, r in bf16
    out = d * 2                                   # o at the activations' dtype
    assert state + ins + out == 133634            # ~133.6 KB
    assert bench.decode_bytes(1, 1, d, d) == 133634
    assert bench.decode_bytes(256, 16, d, d) == 256 * 16 * 133634
    # isotropic, one decay per head: g, omega and b are one value per head
    iso = 2 * (d * d * 4 + 4) + (3 * d + 3) * 2 + d * 2
    assert iso == 132110                          # ~132.1 KB
    assert bench.decode_bytes(1, 1, d, d, variant="iso") == 132110


def test_chunked_flops(bench):
    # 10 C d + 6 d^2 per token-head at C = 64, d = 128
    assert bench.chunk_flops(128, 128) == 180224
    # the FLOP term of the spec roofline stays below the bytes term for the forward
    B, T, H, d = 8, 4096, 16, 128
    flop_s = B * T * H * bench.chunk_flops(d, d) / 2.25e15
    byte_s = bench.fwd_bytes(B, T, H, d, d) / 8e12
    assert flop_s < byte_s


def test_outputs_counted_at_the_input_dtype(bench):
    # o and the gradients count at the activations' dtype (bf16): writing them
    # wider would add bytes to the numerator of the achieved bandwidth, so the
    # default accounting must be the bf16 one
    for fn in (bench.fwd_bytes, bench.bwd_bytes):
        lo = fn(8, 4096, 16, 128, 128, out_bytes=2)
        hi = fn(8, 4096, 16, 128, 128, out_bytes=4)
        assert hi > lo
        assert fn(8, 4096, 16, 128, 128) == lo


def test_job_throughput_sums_ranks(bench):
    # tokens of every rank over the slowest rank's time
    assert bench.job_throughput(1000, 4, 2.0) == pytest.approx(4 * 1000 / 2e-3)


def test_both_arms_report_one_workload(bench):
    cfg = bench.step_config(1)
    assert (cfg["B"], cfg["T"], cfg["H"], cfg["dk"], cfg["dv"]) == (8, 4096, 16, 128, 128)
    assert cfg["activations"] == "bf16" and cfg["outputs"] == "bf16" and cfg["state"] == "f32"
    assert bench.step_config(4)["parallelism"] == "replicas x4"
