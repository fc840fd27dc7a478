// Backward (STE) + fused AdamW kernels, NVFP4, per-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_adamw_nv(int dt, int sub, bool sfpg, const KParams& p, cudaStream_t st)
{
    if (sfpg) return linear_by_dt<1, kBwdSA>(dt, sub, p, st);
    return linear_by_dt<1, kBwdA>(dt, sub, p, st);
}

}  // namespace focus
