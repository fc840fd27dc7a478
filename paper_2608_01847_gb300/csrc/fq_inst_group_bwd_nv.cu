// Group (one launch for several tensors) backward kernels, NVFP4.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_group_bwd_nv(int dt, int sub, bool sfpg, const KGroup& g, cudaStream_t st)
{
    return sfpg ? group_by_dt<1, kBwdS>(dt, sub, g, st) : group_by_dt<1, kBwd>(dt, sub, g, st);
}

}  // namespace focus
