// dpo_step_adan.cu -- fused-step kernel instances for one update rule (see
// dpo_step.cuh); one translation unit per rule so they compile in parallel.
#include "dpo_step.cuh"

namespace dpo {

StepFn pick_step_adan(bool param_bf16, StashKind stash, bool grad_bf16, Correction corr,
                       bool dc, bool pp)
{
    return pick_step<kOptAdan>(param_bf16, stash, grad_bf16, corr, dc, pp);
}

}  // namespace dpo
