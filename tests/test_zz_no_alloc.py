"""pf_lmhead_accept_noalloc against pf_lmhead_accept, through the C ABI.

Callers that cannot allocate device memory where they verify a proposal
(code running during CUDA-graph stream capture, plug-ins whose framework
owns all device memory, allocation-free loops) use the entry point whose
scratch is a fixed array inside the library instead of a workspace they
pass in.  Both run the same kernel, so every output must agree; two calls
in a row also check that the shared array is cleared between calls."""
import numpy as np
import pytest
import torch

from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I
from tests.parity import Case

pytestmark = pytest.mark.gpu


def _clear_outputs(vs):
    for t in (vs.argmax, vs.accept_len, vs.path, vs.out_tokens, vs.last_node):
        t.fill_(-1)
    vs.max_logit.zero_()


def test_noalloc_matches_workspace_entry_point():
    w = I.scaled(I.WORKLOADS["7b-bf16-batch8-paged"], layers=1, prefix=(40, 90), vocab=3000,
                 hidden=256)
    c = Case(w, seed=11)
    vs = c.vs
    vs.lmhead()
    ref = vs.results()
    assert ref["err"] == 0
    for _ in range(2):
        _clear_outputs(vs)
        pb.pf_lmhead_accept_noalloc(vs.lm_desc, torch.cuda.current_stream().cuda_stream)
        got = vs.results()
        assert got["err"] == 0
        for k in ("argmax", "accept_len", "path", "out_tokens", "last_node"):
            np.testing.assert_array_equal(got[k], ref[k])
        np.testing.assert_allclose(got["max_logit"], ref["max_logit"], rtol=0,
                                   atol=2e-3 * (1 + np.abs(ref["max_logit"]).max()))
        c.check_lmhead(got)


def test_noalloc_rejects_more_rows_than_its_scratch_holds():
    d = pb.pf_lm_desc()
    d.dtype, d.batch, d.hidden, d.vocab = pb.PF_BF16, 2, 64, 1000
    d.total_nodes, d.max_nodes = pb.PF_MAX_LM_ROWS + 1, 128
    with pytest.raises(pb.PfError) as e:
        pb.pf_lmhead_accept_noalloc(d, 0)
    assert e.value.status == pb.PF_ERR_SHAPE
    assert "scratch" in pb.pf_last_error()


def test_noalloc_checks_the_descriptor_before_clearing_its_scratch():
    """A descriptor the workspace entry point rejects is rejected with the
    same status, before the scratch is cleared (nothing is queued)."""
    d = pb.pf_lm_desc()
    d.dtype, d.batch, d.hidden, d.vocab = pb.PF_BF16, 1, 64, 1000
    d.total_nodes, d.max_nodes = 4, 4
    fake = 0x10000
    for f in ("cu_nodes", "hidden_states", "tokens", "parent", "argmax", "accept_len", "path",
              "out_tokens"):
        setattr(d, f, fake)
    d.weight = None
    with pytest.raises(pb.PfError) as e:
        pb.pf_lmhead_accept_noalloc(d, 0)
    assert e.value.status == pb.PF_ERR_NULL
