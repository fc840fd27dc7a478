// Forward fake-quantization kernels (every format x dtype x sub-block size).
#include "fq_launch.h"

namespace focus {

cudaError_t launch_fwd(int fmt, int dt, int sub, const KParams& p, cudaStream_t st)
{
    if (fmt == 0) return linear_by_dt<0, kFwd>(dt, sub, p, st);
    return linear_by_dt<1, kFwd>(dt, sub, p, st);
}

}  // namespace focus
