"""Allocation failures injected on the host (dpo_test_fail_allocs): dpo_init
and dpo_muon_init return DPO_ENOMEM with a message, free what they had
allocated before the failing allocation, and leave the library usable."""
from __future__ import annotations

import ctypes

import pytest
import torch

from paper_2606_30634_gb300 import dpo, muon

pytestmark = pytest.mark.gpu


def _free_bytes():
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def test_init_allocation_failures(cuda_device):
    opt = dpo.DelayedAdamW([1000, 77, 4096], device=cuda_device)
    m = muon.DelayedMuon([(256, 512), (300, 700)], device=cuda_device)
    try:
        # dpo_init's one block
        free0 = _free_bytes()
        dpo.dpo_test_fail_allocs(0, 1)
        with pytest.raises(dpo.DpoError) as e:
            dpo.dpo_init(opt.table, opt.param_dtype, opt.stash_dtype, opt.grad_dtype, opt.hp)
        assert e.value.code == dpo.DPO_ENOMEM and "cudaMalloc" in str(e.value)
        assert _free_bytes() == free0
        # dpo_muon_init: the table block, then the workspace (the table freed again)
        L = muon.lib()
        arr = (muon.dpo_matrix * len(m.table))(*m.table)
        for after, what in ((0, "table"), (1, "workspace")):
            dpo.dpo_test_fail_allocs(after, 1)
            out = ctypes.c_void_p()
            rc = L.dpo_muon_init(ctypes.byref(out), arr, len(m.table), m.stash_dtype,
                                 m.grad_dtype, ctypes.byref(m.hp), dpo.DPO_INIT_RESUME, None)
            assert rc == dpo.DPO_ENOMEM and out.value is None
            assert what in L.dpo_muon_last_error(None).decode()
            assert _free_bytes() == free0
        dpo.dpo_test_fail_allocs(0, 0)
        # the hook is off: both kinds of context work on
        opt.step()
        m.step()
        torch.cuda.synchronize()
        assert m.status() == 0
        again = dpo.DelayedAdamW([1000, 77], device=cuda_device)
        again.step()
        again.close()
    finally:
        dpo.dpo_test_fail_allocs(0, 0)
        opt.close()
        m.close()
