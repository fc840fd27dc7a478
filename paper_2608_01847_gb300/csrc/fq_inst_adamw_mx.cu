// Backward (STE) + fused AdamW kernels, MXFP4, per-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_adamw_mx(int dt, int sub, bool sfpg, const KParams& p, cudaStream_t st)
{
    if (sfpg) return dt ? linear_by_sub<0, 1, kBwdSA>(sub, p, st) : linear_by_sub<0, 0, kBwdSA>(sub, p, st);
    return dt ? linear_by_sub<0, 1, kBwdA>(sub, p, st) : linear_by_sub<0, 0, kBwdA>(sub, p, st);
}

}  // namespace focus
