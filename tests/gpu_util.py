"""Helpers of the GPU parity tests: run one verification step through the C ABI
on inputs built by ``synth`` and compare it with the oracle on the same bytes."""

from __future__ import annotations

import torch

import oracle
import paper_2405_00263_gb300 as pkg

ATOL = {torch.float32: 1e-4, torch.bfloat16: 2e-2}


def to_dev(host: dict, dev) -> dict:
    return {k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in host.items()}


def run_gpu(t: dict, scale: float = 0.0, step: pkg.VerifyStep | None = None, **step_kw) -> pkg.VerifyStep:
    B, T, Hq, D = t["q"].shape
    Hkv = t["k_new"].shape[2]
    V = t["logits"].shape[-1]
    if step is None:
        step = pkg.VerifyStep(B, T, Hq, Hkv, D, t["Lcap"], V, t["q"].dtype, device=t["q"].device, **step_kw)
    step.clear_status()
    step.run(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"], t["parent"],
             t["cand"], t["logits"], scale=scale)
    torch.cuda.synchronize()
    return step


def compare_full(host: dict, step: pkg.VerifyStep, t: dict, scale: float = 0.0):
    """Every output against oracle.verify_step (small shapes)."""
    ref = oracle.verify_step(host, scale=scale, typical=step.typical if step.accept == "typical" else None)
    dt = host["q"].dtype
    assert step.device_status() == 0
    err = (step.out.double().cpu() - ref["out"]).abs().max().item()
    assert err <= ATOL[dt], f"attention max-abs {err} > {ATOL[dt]}"
    assert torch.equal(step.argmax.cpu(), ref["argmax"])
    assert torch.equal(step.path.cpu(), ref["path"])
    assert torch.equal(step.accept_len.cpu(), ref["accept_len"])
    assert torch.equal(step.bonus.cpu(), ref["bonus"])
    # the commit and fused schedules record tree nodes, the compaction schedule cache slots
    exp_src = ref["path"] if step.schedule in ("commit", "fused") else ref["src_index"]
    assert torch.equal(step.src_index.cpu(), exp_src)
    assert torch.equal(step.new_cache_len.cpu(), ref["cache_len"])
    kc, vc = t["k_cache"].cpu(), t["v_cache"].cpu()
    for b in range(kc.shape[0]):
        n = int(ref["cache_len"][b])
        assert torch.equal(kc[b, :, :n].view(torch.int16 if dt == torch.bfloat16 else torch.int32),
                           ref["k_cache"][b, :, :n].view(torch.int16 if dt == torch.bfloat16 else torch.int32))
        assert torch.equal(vc[b, :, :n].view(torch.int16 if dt == torch.bfloat16 else torch.int32),
                           ref["v_cache"][b, :, :n].view(torch.int16 if dt == torch.bfloat16 else torch.int32))
    return err, ref
