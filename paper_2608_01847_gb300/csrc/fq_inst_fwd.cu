// Forward fake-quantization kernels (every format x dtype x sub-block size).
#include "fq_launch.h"

namespace focus {

cudaError_t launch_fwd(int fmt, int dt, int sub, const KParams& p, cudaStream_t st)
{
    if (fmt == 0) return dt ? linear_by_sub<0, 1, kFwd>(sub, p, st) : linear_by_sub<0, 0, kFwd>(sub, p, st);
    return dt ? linear_by_sub<1, 1, kFwd>(sub, p, st) : linear_by_sub<1, 0, kFwd>(sub, p, st);
}

}  // namespace focus
