// fq_noalloc.cu -- the NVFP4 per-tensor alpha pass without caller-provided
// scratch, for callers that cannot allocate device memory.
//
// focus_nvfp4_alpha needs a scratch buffer of per-CTA partial maxima, which
// the caller normally allocates.  Some callers cannot: a plugin running
// inside a host application that owns every device allocation and hands the
// plugin only its input and output buffers, or a latency-bound loop that must
// never reach cudaMalloc (which can synchronise the whole device).  For them
// this file keeps the partials in a fixed array in the library's own device
// memory instead.
//
// The array below is a file-scope __device__ variable: every GPU that loads
// this library holds its 16 KiB until the process exits.  Host code cannot
// use its name as an address (on the host the name is a stand-in, not a
// device pointer), so the device address is looked up with
// cudaGetSymbolAddress once per device, with that device current, the first
// time the entry point runs there.
#include <cstdint>
#include <cstring>
#include <mutex>

#include "../../include/focus_fq.h"
#include "fq_launch.h"

#define FOCUS_API extern "C" __attribute__((visibility("default")))

namespace focus {
namespace {

// Largest number of per-CTA partial maxima the static scratch holds: 4096
// fp32 values (16 KiB), enough for the alpha pass's grid on any GPU with up
// to 512 SMs (it launches at most 8 CTAs per SM).
constexpr uint32_t kStaticAlphaPartials = 4096;

__device__ __align__(256) float g_alpha_partials[kStaticAlphaPartials];

constexpr int kMaxDevices = 64;
float* g_partials_addr[kMaxDevices] = {nullptr};
std::mutex g_setup_mutex;

// Device address of g_alpha_partials on the current device (looked up once
// per device, with that device current, and kept for the life of the
// process: it is not valid across a reset of the device's context).
int static_partials(float** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return FOCUS_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return FOCUS_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_partials_addr[dev] == nullptr) {
        void* addr = nullptr;
        if (cudaGetSymbolAddress(&addr, g_alpha_partials) != cudaSuccess || addr == nullptr)
            return FOCUS_ERR_CUDA;
        g_partials_addr[dev] = static_cast<float*>(addr);
    }
    *out = g_partials_addr[dev];
    return FOCUS_OK;
}

bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }

}  // namespace
}  // namespace focus

using namespace focus;

FOCUS_API int focus_nvfp4_alpha_noalloc(const focus_desc_t* desc, const void* x,
                                        float* alpha_out, focus_stream_t stream)
{
    // same shape rules as focus_nvfp4_alpha (only the tensor shape is used)
    if (!desc) return FOCUS_ERR_INVALID_ARG;
    if (desc->rows < 0 || desc->cols < 0 || desc->ld < desc->cols) return FOCUS_ERR_INVALID_ARG;
    if (desc->dtype != FOCUS_F32 && desc->dtype != FOCUS_BF16 && desc->dtype != FOCUS_F16)
        return FOCUS_ERR_INVALID_ARG;
    if (desc->cols % 8 != 0) return FOCUS_ERR_INVALID_ARG;
    if ((desc->ld * (desc->dtype == FOCUS_F32 ? 4 : 2)) % 16 != 0) return FOCUS_ERR_MISALIGNED;
    if (desc->rows > 0 && desc->cols > 0 && desc->rows > ((int64_t(1) << 31) - 1) / (desc->cols / 8))
        return FOCUS_ERR_UNSUPPORTED;
    const bool empty = desc->rows == 0 || desc->cols == 0;
    if (!alpha_out || (!empty && !x)) return FOCUS_ERR_INVALID_ARG;
    if (misaligned(x, 16) || misaligned(alpha_out, 4)) return FOCUS_ERR_MISALIGNED;

    KParams p;
    std::memset(&p, 0, sizeof(p));
    p.x = x;
    p.ld = static_cast<uint64_t>(desc->ld);
    p.cpr = static_cast<uint32_t>(desc->cols / 8);
    p.rows = static_cast<uint32_t>(desc->rows);
    p.n_chunks = static_cast<uint32_t>(desc->rows * (desc->cols / 8));
    p.div_cpr = make_fastdiv(p.cpr > 0 ? p.cpr : 1u);
    p.strided = desc->ld != desc->cols;

    // The partial pass needs one slot per CTA; refuse a grid the array cannot hold.
    if (alpha_grid(p.n_chunks) > kStaticAlphaPartials) return FOCUS_ERR_WORKSPACE;
    float* partials = nullptr;
    const int rc = static_partials(&partials);
    if (rc != FOCUS_OK) return rc;
    // Nothing in the array has to start at zero: every slot the final
    // reduction reads is written by its CTA earlier in the same call.
    p.ws = partials;
    return launch_alpha(desc->dtype, p, alpha_out, reinterpret_cast<cudaStream_t>(stream)) ==
                   cudaSuccess
               ? FOCUS_OK
               : FOCUS_ERR_CUDA;
}
