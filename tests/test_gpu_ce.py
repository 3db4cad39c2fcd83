"""GPU parity of the reduced-vocabulary LM-head cross entropy with logits
masking (through the C ABI) against the fp64 oracle on the same seeded bf16
inputs.  J and the trainable positions are integer work: compared exactly.
Tolerances: loss relative 1e-4 (fp32 logits and fp32 log-sum-exp; derived
from fp32 rounding of d-term dot products and of the exp / log calls,
~1e-6 relative per logit), per-position losses absolute 1e-3, dh relative
Frobenius 5e-3 (softmax - onehot enters the contraction in bf16 and dh is
rounded to bf16, unit roundoff 2^-9)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_19528_gb300 import lora, synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

TOL_LOSS = 1e-4
TOL_TOKEN = 1e-3
TOL_DH = 5e-3


class CeCase:
    def __init__(self, T, d, V, k=None, frac=0.3, cluster=64, cfg=40, seed=0, table_width=None):
        self.T, self.d, self.V, self.k = T, d, V, k
        self.h_bits = synth.gen_h(seed, cfg, T, d)
        self.E_bits = synth.gen_E(seed, cfg, V, d)
        self.targets = synth.gen_targets(seed, cfg, T, V, cluster)
        self.mask = synth.gen_mask(T, frac)
        self.topk = None if k is None else synth.gen_topk_table(seed, cfg, V, table_width or k, cluster)
        dev = "cuda"
        self.h, self.E = G.dev_bf16(self.h_bits), G.dev_bf16(self.E_bits)
        self.t_targets = torch.from_numpy(self.targets).to(dev)
        self.t_mask = torch.from_numpy(self.mask).to(dev)
        self.t_topk = None if self.topk is None else torch.from_numpy(self.topk).to(dev)
        self.loss = torch.full((1,), float("nan"), device=dev)
        self.token_loss = torch.full((T,), float("nan"), device=dev)
        self.dh = torch.full((T, d), float("nan"), dtype=torch.bfloat16, device=dev)
        self.vocab = torch.full((V,), -1, dtype=torch.int32, device=dev)

    def args(self, mask=True):
        return lora.make_ce_args(self.T, self.d, self.V, self.h, self.E, self.t_targets, self.loss,
                                 mask=self.t_mask if mask else None, topk=self.t_topk,
                                 ld_topk=0 if self.topk is None else self.topk.shape[1], k=self.k or 0,
                                 token_loss=self.token_loss, dh=self.dh, vocab=self.vocab)

    def run(self, mask=True):
        a = self.args(mask)
        ws = G.workspace(lora.lora_ce_workspace_size(a))
        counts = lora.lora_ce_fwd_bwd(a, ws, ws.numel())
        torch.cuda.synchronize()
        assert lora.lora_read_status() == lora.LORA_OK
        return counts

    def oracle(self, mask=True):
        m = self.mask.astype(bool) if mask else np.ones(self.T, dtype=bool)
        J = np.arange(self.V) if self.topk is None else oracle.reduced_vocab(self.targets, m, self.topk, self.k)
        h = synth.bf16_bits_to_f64(self.h_bits)
        E = synth.bf16_bits_to_f64(self.E_bits)
        loss, per, dh = oracle.ce_forward_backward(h, E, self.targets, m, J)
        return J, loss, per, dh, int(m.sum())


def check(case, mask=True):
    nT, nJ = case.run(mask)
    J, loss, per, dh, nT_want = case.oracle(mask)
    assert nT == nT_want and nJ == len(J), (nT, nJ, nT_want, len(J))
    got_J = case.vocab[:nJ].cpu().numpy()
    assert np.array_equal(got_J, J.astype(np.int32)), "reduced vocabulary differs"
    got_loss = float(case.loss.item())
    assert abs(got_loss - loss) <= TOL_LOSS * abs(loss), (got_loss, loss)
    got_per = case.token_loss.double().cpu().numpy()
    assert np.abs(got_per - per).max() <= TOL_TOKEN, np.abs(got_per - per).max()
    got_dh = G.host_f64(case.dh)
    assert G.rel_fro(got_dh, dh) <= TOL_DH, G.rel_fro(got_dh, dh)
    off = ~(case.mask.astype(bool) if mask else np.ones(case.T, dtype=bool))
    assert np.all(got_dh[off] == 0.0), "dh of a non-trainable position must be exactly zero"
    return nT, nJ


# the last case has few output tiles over a deep contraction (d = 3072): the
# logits contraction is split and its log-sum-exp partials come from the split
# reduce instead of the epilogue
@pytest.mark.parametrize("T,d,V,k", [(300, 256, 5000, 37), (128, 512, 3000, 200), (1000, 1024, 20000, 64),
                                     (128, 3072, 20000, 64)],
                         ids=["T300_d256_V5000_k37", "T128_d512_V3000_k200", "T1000_d1024_V20000_k64",
                              "T128_d3072_V20000_k64_split"])
def test_ce_topk_parity(T, d, V, k):
    case = CeCase(T, d, V, k=k, table_width=k + 3)
    nT, nJ = check(case)
    assert 0 < nJ < V


def test_ce_full_vocab_parity():
    case = CeCase(256, 256, 4000, k=None, frac=0.5)
    nT, nJ = check(case)
    assert nJ == 4000


def test_ce_table_covering_the_whole_vocabulary():
    """A top-k table whose rows cover every token makes J the whole
    vocabulary: E is read in place although a table was given."""
    case = CeCase(128, 256, 600, k=600, frac=0.5)
    nT, nJ = check(case)
    assert nJ == 600


def test_ce_logits_masking_identity():
    """Full vocabulary: the logits and losses of a trainable position do not
    depend on which other positions are trainable, so the masked call's
    per-position losses and dh rows equal those of the call with every
    position trainable, bit for bit (the paper: logits masking gives identical
    losses and gradients)."""
    case = CeCase(264, 256, 3000, k=None, frac=0.4)
    case.run(mask=True)
    tl_m, dh_m = case.token_loss.clone(), case.dh.clone()
    case.run(mask=False)
    m = torch.from_numpy(case.mask.astype(bool)).to("cuda")
    assert torch.equal(tl_m[m], case.token_loss[m])
    assert torch.equal(dh_m[m].view(torch.int16), case.dh[m].view(torch.int16))
    assert torch.all(tl_m[~m] == 0) and torch.all(dh_m[~m] == 0)


def test_ce_no_trainable_positions():
    case = CeCase(64, 256, 1000, k=16, frac=0.0)
    nT, nJ = case.run()
    assert nT == 0 and nJ == 0
    assert float(case.loss.item()) == 0.0
    assert torch.all(case.token_loss == 0) and torch.all(case.dh == 0)


def test_ce_bad_input():
    case = CeCase(64, 256, 1000, k=16, frac=1.0)
    case.t_targets[5] = 1000  # out of the vocabulary
    a = case.args()
    ws = G.workspace(lora.lora_ce_workspace_size(a))
    with pytest.raises(lora.LoraError) as e:
        lora.lora_ce_fwd_bwd(a, ws, ws.numel())
    assert e.value.code == lora.LORA_EINVAL
    torch.cuda.synchronize()
    assert torch.isnan(case.loss).all() and torch.isnan(case.dh).all(), "outputs must be untouched"
