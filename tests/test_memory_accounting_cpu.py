"""Memory sanity of the byte accounting against the paper's Table efficiency_memory
(tests/golden/memory_qwen3_30b.txt): the FP16 size of the Qwen3-30B-A3B MoE stack
reproduces the printed 54.00 (GiB), and the stored size of the synthetic 2.0-bit workload
(codes at their bit-widths, fp16 scale + zero per group, fp32 alpha per live unit, bf16
bases) comes within a few percent of the printed BitsMoE figure.  The workload's bits
stand in for the paper's allocation, so this checks the accounting, not parity."""
import os

import numpy as np

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden():
    out = {}
    with open(os.path.join(GOLDEN, "memory_qwen3_30b.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                out[k] = float(v)
    return out


def test_fp16_stack_size_is_the_printed_figure():
    ref = _golden()
    layers, E, D, I = 48, 128, 2048, 768
    assert abs(layers * E * 3 * D * I * 2 / 2 ** 30 - ref["fp16"]) < 0.005


def test_stored_two_bit_stack_is_near_the_printed_figure():
    ref = _golden()
    spec = synth.WORKLOADS["qw3"]
    layer = synth.make_layer(spec, seed=0)
    bits = layer["bits"].astype(np.int64)
    live = bits > 0
    quant = live & (bits < 16)
    ng = spec.I // spec.group
    per_layer = (3 * spec.D * spec.n * 2                      # bf16 bases
                 + int((bits * spec.I).sum()) // 8             # codes at their bit-widths
                 + int(quant.sum()) * ng * 4                   # fp16 scale + zero per group
                 + int(live.sum()) * 4)                        # fp32 alpha per live unit
    got = 48 * per_layer / 2 ** 30
    assert abs(got - ref["bitsmoe_2bit"]) / ref["bitsmoe_2bit"] < 0.05, got
