// Export (pack) kernels and the NVFP4 per-tensor alpha pass.
#include "fq_launch.h"

namespace focus {

// One CTA: max of the per-CTA partial maxima, alpha = fl(amax / 2688) (Eq. 2).
__device__ __forceinline__ void alpha_final_kernel_body(const float* partials, uint32_t n, float* alpha_out)
{
    __shared__ float red[kThreads / 32];
    float m = 0.0f;
    for (uint32_t i = threadIdx.x; i < n; i += kThreads) m = fmaxf(m, partials[i]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFullMask, m, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x < 32) {
        m = (threadIdx.x < kThreads / 32) ? red[threadIdx.x] : 0.0f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFullMask, m, o));
        if (threadIdx.x == 0) *alpha_out = __fdiv_rn(m, 2688.0f);  // M_FP4 * M_FP8
    }
}

__global__ void __launch_bounds__(kThreads) alpha_final_kernel(const float* partials, uint32_t n,
                                                               float* alpha_out)
{
    // launched early behind the partial pass: wait until it has completed
    // and its partials are visible (a no-op without that dependency)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    alpha_final_kernel_body(partials, n, alpha_out);
}

cudaError_t launch_pack(int fmt, int dt, int sub, const KParams& p, cudaStream_t st)
{
    if (fmt == 0) return linear_by_dt<0, kPack>(dt, sub, p, st);
    return linear_by_dt<1, kPack>(dt, sub, p, st);
}

// Group form: CTA t reduces the partials of tensor t to alpha_out[t].
__global__ void __launch_bounds__(kThreads) alpha_group_final_kernel(const __grid_constant__ KGroup g,
                                                                     float* alpha_out)
{
    const uint32_t t = blockIdx.x;
    alpha_final_kernel_body(g.p[0].ws + g.start[t], g.start[t + 1] - g.start[t], alpha_out + t);
}

cudaError_t launch_alpha_group(int dt, const KGroup& g, float* alpha_out, cudaStream_t st)
{
    const uint32_t grid = g.start[g.n];
    if (grid > 0) {
        if (dt == 1) alpha_group_partial_kernel<1><<<grid, kThreads, 0, st>>>(g);
        else if (dt == 2) alpha_group_partial_kernel<2><<<grid, kThreads, 0, st>>>(g);
        else alpha_group_partial_kernel<0><<<grid, kThreads, 0, st>>>(g);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    alpha_group_final_kernel<<<g.n, kThreads, 0, st>>>(g, alpha_out);
    return cudaGetLastError();
}

cudaError_t launch_alpha(int dt, const KParams& p, float* alpha_out, cudaStream_t st)
{
    const uint32_t grid = alpha_grid(p.n_chunks);
    if (p.n_chunks > 0) {
        if (dt == 1) alpha_partial_kernel<1><<<grid, kThreads, 0, st>>>(p);
        else if (dt == 2) alpha_partial_kernel<2><<<grid, kThreads, 0, st>>>(p);
        else alpha_partial_kernel<0><<<grid, kThreads, 0, st>>>(p);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    // programmatic dependent launch: the one-CTA reduction is scheduled while
    // the partial pass still runs, instead of after it
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(kThreads);
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = p.n_chunks > 0 ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, alpha_final_kernel, static_cast<const float*>(p.ws),
                              p.n_chunks > 0 ? grid : 0u, alpha_out);
}

}  // namespace focus
