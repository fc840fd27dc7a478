// Group (one launch for several tensors) forward kernels, both formats.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_group_fwd(int fmt, int dt, int sub, const KGroup& g, cudaStream_t st)
{
    return fmt == 0 ? group_by_dt<0, kFwd>(dt, sub, g, st) : group_by_dt<1, kFwd>(dt, sub, g, st);
}

}  // namespace focus
