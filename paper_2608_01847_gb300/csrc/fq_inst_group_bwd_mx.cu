// Group (one launch for several tensors) backward kernels, MXFP4.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_group_bwd_mx(int dt, int sub, bool sfpg, const KGroup& g, cudaStream_t st)
{
    return sfpg ? group_by_dt<0, kBwdS>(dt, sub, g, st) : group_by_dt<0, kBwd>(dt, sub, g, st);
}

}  // namespace focus
