"""GPU tests of the top-k similarity table (through the C ABI) against the
oracle.  The table is integer output decided by floating point: the oracle
reproduces the library's normalised bf16 embedding exactly and decides on
exact similarities of it, while the tensor cores sum the d exact products in
fp32, within eps = 2 d 2^-24 of the exact value (unit vectors).  So a row is
checked for what is unique -- every token whose exact similarity exceeds the
exact k-th largest by more than 2 eps is present, the first entry is the
token itself -- and for validity: k distinct tokens, in descending exact
similarity up to 2 eps, none outside missing by more than 2 eps.  Small
exact cases (a hand-worked table with ties) must match exactly."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2606_19528_gb300 import lora, synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def run_table(bits, k):
    V, d = bits.shape
    E = G.dev_bf16(bits)
    table = torch.full((V, k), -1, dtype=torch.int32, device="cuda")
    ws = G.workspace(lora.lora_topk_workspace_size(V, d, k))
    lora.lora_topk_table(E, V, d, k, table, ws, ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK
    return table.cpu().numpy()


def test_topk_handworked_exact():
    with open(os.path.join(GOLDEN, "topk_table_handworked_V4_d2.json")) as f:
        g = json.load(f)
    for E, want in ((g["E"], g["table_k4"]), (g["ties"]["E"], g["ties"]["table_k4"])):
        x = np.zeros((4, 8))
        x[:, :2] = np.array(E, dtype=np.float64)  # d padded to 8 with zeros: norms and products unchanged
        got = run_table(synth.to_bf16_bits(x), 4)
        assert got.tolist() == want, (got.tolist(), want)


def check_rows(bits, table, k, rows):
    V, d = bits.shape
    eps = 2.0 * d * 2.0 ** -24
    En = oracle.normalize_rows(bits)
    C = oracle.similarities(En, rows)
    for r, i in enumerate(rows):
        L = table[i]
        assert len(set(L.tolist())) == k and L.min() >= 0 and L.max() < V, i
        assert L[0] == i, (i, L[:4])
        c = C[r]
        cl = c[L]
        assert np.all(cl[:-1] >= cl[1:] - 2 * eps), i
        kth = np.sort(c)[::-1][k - 1]
        outside = np.ones(V, dtype=bool)
        outside[L] = False
        assert np.all(c[outside] <= cl[-1] + 2 * eps), i
        must = np.nonzero(c > kth + 2 * eps)[0]
        assert np.all(np.isin(must, L)), i


# V >= 32768 takes the sampled-threshold selection, smaller V the radix path
@pytest.mark.parametrize("V,d,k", [(5000, 256, 37), (1200, 64, 1024), (20000, 1024, 500), (32767, 64, 64),
                                   (32768, 64, 64), (40000, 64, 300), (70000, 128, 1024)],
                         ids=["V5000_d256_k37", "V1200_d64_k1024", "V20000_d1024_k500", "V32767_d64_k64",
                              "V32768_d64_k64_sampled", "V40000_d64_k300_sampled", "V70000_d128_k1024_sampled"])
def test_topk_table_parity(V, d, k):
    bits = synth.gen_E(0, 50, V, d)
    table = run_table(bits, k)
    rng = np.random.default_rng(V)
    rows = np.unique(np.concatenate([[0, V - 1, 511, 512], rng.integers(0, V, 60)]))
    check_rows(bits, table, k, rows)


def test_topk_argument_errors():
    with pytest.raises(lora.LoraError) as e:
        lora.lora_topk_workspace_size(100, 12, 5)  # d not a multiple of 8
    assert e.value.code == lora.LORA_EINVAL
    with pytest.raises(lora.LoraError) as e:
        lora.lora_topk_workspace_size(100, 16, 101)  # k > V
    assert e.value.code == lora.LORA_EINVAL
    with pytest.raises(lora.LoraError) as e:
        lora.lora_topk_workspace_size(5000, 16, 1025)  # k beyond the selection's capacity
    assert e.value.code == lora.LORA_EINVAL


def test_topk_sampled_ties_and_fallback():
    """Rows 0..1999 are one vector u, rows 2000..4999 one vector v with
    cos(u, v) about 0.9, the rest random (V = 40000, k = 1000).  A u row's
    sampled threshold lands on v's similarity, so 5000 values pass it (more
    than the 4096 candidate slots) and the row falls back to the radix select;
    a v row passes 3000 tied values and stays on the sampled path.  Identical
    inputs give identical tensor-core sums, so the ties are exact and the
    lower index goes first: u rows list tokens 0..999, v rows 2000..2999."""
    V, d, k = 40000, 64, 1000
    bits = synth.gen_E(0, 51, V, d)
    x = synth.bf16_bits_to_f64(bits)
    u = x[7] / np.linalg.norm(x[7])
    w = x[11] - (x[11] @ u) * u
    v = 0.9 * u + np.sqrt(1 - 0.81) * w / np.linalg.norm(w)
    ub, vb = synth.to_bf16_bits(u[None, :]), synth.to_bf16_bits(v[None, :])
    bits = bits.copy()
    bits[0:2000] = ub
    bits[2000:5000] = vb
    table = run_table(bits, k)
    for i in (0, 1, 1999):
        assert table[i].tolist() == list(range(1000)), i
    for i in (2000, 4999):
        assert table[i].tolist() == list(range(2000, 3000)), i
    check_rows(bits, table, k, np.array([5000, 12345, V - 1]))
