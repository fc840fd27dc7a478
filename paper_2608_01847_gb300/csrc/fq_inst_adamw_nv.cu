// Backward (STE) + fused AdamW kernels, NVFP4, per-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_adamw_nv(int dt, int sub, bool sfpg, const KParams& p, cudaStream_t st)
{
    if (sfpg) return dt ? linear_by_sub<1, 1, kBwdSA>(sub, p, st) : linear_by_sub<1, 0, kBwdSA>(sub, p, st);
    return dt ? linear_by_sub<1, 1, kBwdA>(sub, p, st) : linear_by_sub<1, 0, kBwdA>(sub, p, st);
}

}  // namespace focus
