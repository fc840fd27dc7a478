// fq_abi.cu -- the extern "C" entry points declared in include/focus_fq.h:
// argument validation, launch parameters, scratch sizing, error mapping.
// No allocation, no host synchronisation, no exception crosses the ABI.
#include <algorithm>
#include <cstdint>
#include <cstring>

#include "../../include/focus_fq.h"
#include "fq_launch.h"

#define FOCUS_API extern "C" __attribute__((visibility("default")))

namespace focus {

cudaError_t launch_bwd_mx(int dt, int sub, const KParams& p, cudaStream_t st);
cudaError_t launch_bwd_nv(int dt, int sub, const KParams& p, cudaStream_t st);
cudaError_t launch_bwd_shared_mx(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st);
cudaError_t launch_bwd_shared_nv(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st);

int shared_bwd_occupancy_mx(int dt, int sub);
int shared_bwd_occupancy_nv(int dt, int sub);

int shared_bwd_occupancy(int fmt, int dt, int sub)
{
    return fmt == 0 ? shared_bwd_occupancy_mx(dt, sub) : shared_bwd_occupancy_nv(dt, sub);
}

cudaError_t launch_bwd(int fmt, int dt, int sub, const KParams& p, cudaStream_t st)
{
    return fmt == 0 ? launch_bwd_mx(dt, sub, p, st) : launch_bwd_nv(dt, sub, p, st);
}

cudaError_t launch_bwd_shared(int fmt, int dt, int sub, const KParams& p, uint32_t ny,
                              cudaStream_t st)
{
    return fmt == 0 ? launch_bwd_shared_mx(dt, sub, p, ny, st)
                    : launch_bwd_shared_nv(dt, sub, p, ny, st);
}

namespace {

constexpr int64_t kMaxChunks = (int64_t(1) << 31) - 1;

bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }

// Shape checks common to every entry point; `method` adds the format,
// block and sub-block rules (the alpha pass needs only the tensor shape).
int check_desc(const focus_desc_t* d, bool method)
{
    if (!d) return FOCUS_ERR_INVALID_ARG;
    if (d->rows < 0 || d->cols < 0 || d->ld < d->cols || d->ld < 0) return FOCUS_ERR_INVALID_ARG;
    if (d->dtype != FOCUS_F32 && d->dtype != FOCUS_BF16 && d->dtype != FOCUS_F16) return FOCUS_ERR_INVALID_ARG;
    if (d->cols % 8 != 0) return FOCUS_ERR_INVALID_ARG;
    // rows start on 16-byte boundaries (128-bit accesses; 256-bit ones when
    // every row of every array starts on a 32-byte boundary)
    if ((d->ld * (d->dtype == FOCUS_F32 ? 4 : 2)) % 16 != 0) return FOCUS_ERR_MISALIGNED;
    if (d->rows > 0 && d->cols > 0 && d->rows > kMaxChunks / (d->cols / 8)) return FOCUS_ERR_UNSUPPORTED;
    if (!method) return FOCUS_OK;
    if (d->fmt != FOCUS_MXFP4 && d->fmt != FOCUS_NVFP4) return FOCUS_ERR_INVALID_ARG;
    if (d->ste != FOCUS_STE_IDENTITY && d->ste != FOCUS_STE_CLIPPED) return FOCUS_ERR_INVALID_ARG;
    if (d->mx_rule != FOCUS_MX_CEIL && d->mx_rule != FOCUS_MX_FLOOR) return FOCUS_ERR_INVALID_ARG;
    if (d->coef_shared_rows != 0 && d->coef_shared_rows != 1) return FOCUS_ERR_INVALID_ARG;
    const int B = d->fmt == FOCUS_MXFP4 ? 32 : 16;
    if (d->block != B) return FOCUS_ERR_UNSUPPORTED;
    const int b = d->sub_block;
    if (b != 2 && b != 4 && b != 8 && b != 16 && b != 32) return FOCUS_ERR_UNSUPPORTED;
    if (b > B || B % b != 0) return FOCUS_ERR_UNSUPPORTED;
    if (d->cols % B != 0) return FOCUS_ERR_INVALID_ARG;
    return FOCUS_OK;
}

KParams make_params(const focus_desc_t* d)
{
    KParams p;
    std::memset(&p, 0, sizeof(p));
    p.ld = static_cast<uint64_t>(d->ld);
    p.cpr = static_cast<uint32_t>(d->cols / 8);
    p.rows = static_cast<uint32_t>(d->rows);
    p.n_chunks = static_cast<uint32_t>(d->rows * (d->cols / 8));
    p.div_cpr = make_fastdiv(p.cpr > 0 ? p.cpr : 1u);
    const int B = d->fmt == FOCUS_NVFP4 ? 16 : 32;
    p.bpr = static_cast<uint32_t>(d->cols / B);
    p.n_blocks = static_cast<uint32_t>(d->rows * (d->cols / B));
    p.div_bpr = make_fastdiv(p.bpr > 0 ? p.bpr : 1u);
    p.tx = shared_tx(p.bpr);
    p.strided = d->ld != d->cols;
    p.shared = d->coef_shared_rows;
    p.ste = d->ste;
    p.mx_rule = d->mx_rule;
    return p;
}

int map_cuda(cudaError_t e) { return e == cudaSuccess ? FOCUS_OK : FOCUS_ERR_CUDA; }

// The element arrays of a call (x, y, g, gx; NULL ones ignored) must start
// on 16-byte boundaries; the kernels take 256-bit accesses when every row of
// every one of them starts on a 32-byte boundary, else two 128-bit ones.
bool rows_misaligned(const void* a, const void* b, const void* c)
{
    return misaligned(a, 16) || misaligned(b, 16) || misaligned(c, 16);
}

int rows_half(const focus_desc_t* d, const void* a, const void* b, const void* c)
{
    const bool pitch32 = (d->ld * (d->dtype == FOCUS_F32 ? 4 : 2)) % 32 == 0;
    return (!pitch32 || misaligned(a, 32) || misaligned(b, 32) || misaligned(c, 32)) ? 1 : 0;
}

// Sub-block size the kernels run with: without DGS coefficients (and without
// their gradient) every sub-block of a block shares S^q, so one sub-block per
// block gives identical results.
int effective_sub(const focus_desc_t* d, const float* dgs, const float* gdgs)
{
    return (dgs == nullptr && gdgs == nullptr) ? d->block : d->sub_block;
}

int check_coef_ptrs(const float* a, const float* b, const float* c, const float* e)
{
    if (misaligned(a, 16) || misaligned(b, 16) || misaligned(c, 16) || misaligned(e, 16))
        return FOCUS_ERR_MISALIGNED;
    return FOCUS_OK;
}

size_t bwd_ws_bytes(const focus_desc_t* d);

// Row groups of the shared-row backward for a descriptor: a function of the
// descriptor and the device only (the occupancy of the kernel for the
// descriptor's sub-block size), so the workspace query and the launch agree;
// a call without DGS runs the block-sized sub-block kernel with the same row
// groups, whose partials then fit in less of the workspace.
uint32_t shared_groups(const focus_desc_t* d)
{
    const uint32_t bpr = static_cast<uint32_t>(d->cols / d->block);
    return shared_row_groups(static_cast<uint32_t>(d->rows), bpr,
                             shared_bwd_occupancy(d->fmt, d->dtype, d->sub_block));
}

// Bytes of the scale tiles of the MMA layout: 128-row x 4-column tiles of
// the [rows, cols/block] scale matrix, 512 bytes each.
size_t mma_scale_bytes(const focus_desc_t* d)
{
    const int64_t sc = d->cols / d->block;
    return static_cast<size_t>((d->rows + 127) / 128) * static_cast<size_t>((sc + 3) / 4) * 512;
}

// Column finalisation of the shared-row backward alone (no rows to reduce).
cudaError_t launch_shared_finalize(int fmt, int sub, const KParams& p, cudaStream_t st)
{
    if (fmt == 0) {
        switch (sub) {
        case 2: return run_shared_finalize<0, 2>(p, 0, st);
        case 4: return run_shared_finalize<0, 4>(p, 0, st);
        case 8: return run_shared_finalize<0, 8>(p, 0, st);
        case 16: return run_shared_finalize<0, 16>(p, 0, st);
        case 32: return run_shared_finalize<0, 32>(p, 0, st);
        default: break;
        }
    } else {
        switch (sub) {
        case 2: return run_shared_finalize<1, 2>(p, 0, st);
        case 4: return run_shared_finalize<1, 4>(p, 0, st);
        case 8: return run_shared_finalize<1, 8>(p, 0, st);
        case 16: return run_shared_finalize<1, 16>(p, 0, st);
        default: break;
        }
    }
    return cudaErrorInvalidValue;
}

// The fused optimizer's arguments (null `hp` for the plain backward).
struct OptArgs {
    float* crs;
    float* dgs;
    float* sfp;
    const focus_adamw_t* hp;
    const focus_adamw_state_t* state;
    const int64_t* step;
};

bool finite_ge0(float v) { return v >= 0.0f && v <= 3.4028234663852886e38f; }

int check_opt(const OptArgs& o)
{
    if (!o.hp || !o.state || !o.step) return FOCUS_ERR_INVALID_ARG;
    const focus_adamw_t& h = *o.hp;
    if (!finite_ge0(h.lr_coef) || !finite_ge0(h.lr_scale) || !finite_ge0(h.weight_decay))
        return FOCUS_ERR_INVALID_ARG;
    if (!(h.beta1 >= 0.0f && h.beta1 < 1.0f) || !(h.beta2 >= 0.0f && h.beta2 < 1.0f))
        return FOCUS_ERR_INVALID_ARG;
    if (!(finite_ge0(h.eps) && h.eps > 0.0f)) return FOCUS_ERR_INVALID_ARG;
    const focus_adamw_state_t& s = *o.state;
    if ((o.crs && (!s.m_crs || !s.v_crs)) || (o.dgs && (!s.m_dgs || !s.v_dgs)) ||
        (o.sfp && (!s.m_sfp || !s.v_sfp)))
        return FOCUS_ERR_INVALID_ARG;
    if (misaligned(o.step, 8)) return FOCUS_ERR_MISALIGNED;
    if (o.crs && (misaligned(s.m_crs, 16) || misaligned(s.v_crs, 16))) return FOCUS_ERR_MISALIGNED;
    if (o.dgs && (misaligned(s.m_dgs, 16) || misaligned(s.v_dgs, 16))) return FOCUS_ERR_MISALIGNED;
    if (o.sfp && (misaligned(s.m_sfp, 16) || misaligned(s.v_sfp, 16))) return FOCUS_ERR_MISALIGNED;
    return FOCUS_OK;
}

void set_opt(KParams& p, const OptArgs& o)
{
    const focus_adamw_t& h = *o.hp;
    p.new_crs = o.crs;
    p.new_dgs = o.dgs;
    p.new_sfp = o.sfp;
    p.opt_m[0] = o.crs ? o.state->m_crs : nullptr;
    p.opt_v[0] = o.crs ? o.state->v_crs : nullptr;
    p.opt_m[1] = o.dgs ? o.state->m_dgs : nullptr;
    p.opt_v[1] = o.dgs ? o.state->v_dgs : nullptr;
    p.opt_m[2] = o.sfp ? o.state->m_sfp : nullptr;
    p.opt_v[2] = o.sfp ? o.state->v_sfp : nullptr;
    p.step = reinterpret_cast<const long long*>(o.step);
    p.lr_c = h.lr_coef;
    p.lr_s = h.lr_scale;
    p.beta1 = h.beta1;
    p.beta2 = h.beta2;
    p.eps = h.eps;
    p.decay_c = static_cast<float>(1.0 - static_cast<double>(h.lr_coef) * h.weight_decay);
    p.decay_s = static_cast<float>(1.0 - static_cast<double>(h.lr_scale) * h.weight_decay);
}

// The backward with or without the fused optimizer step.
int run_bwd(const focus_desc_t* desc, const void* x, const float* crs, const float* dgs,
            const float* alpha, const float* sfp, const void* g, void* gx, float* gcrs,
            float* gdgs, float* gsfp, void* ws, size_t ws_bytes, cudaStream_t st,
            const OptArgs* opt)
{
    int rc = check_desc(desc, true);
    if (rc) return rc;
    if ((sfp || gsfp) && desc->coef_shared_rows) return FOCUS_ERR_INVALID_ARG;
    if (opt && (rc = check_opt(*opt))) return rc;
    const bool learn = opt && (opt->crs || opt->dgs || opt->sfp);
    const bool want_T = gcrs != nullptr || gdgs != nullptr || (learn && (crs || dgs));
    if (rows_misaligned(x, g, gx) || misaligned(alpha, 4) || misaligned(sfp, 4) || misaligned(gsfp, 4))
        return FOCUS_ERR_MISALIGNED;
    if ((rc = check_coef_ptrs(crs, dgs, gcrs, gdgs))) return rc;
    KParams p = make_params(desc);
    p.half = rows_half(desc, x, g, gx);
    p.x = x;
    p.g = g;
    p.gx = gx;
    p.crs = crs;
    p.dgs = dgs;
    p.alpha = alpha;
    p.sfp = sfp;
    p.gcrs = gcrs;
    p.gdgs = gdgs;
    p.gsfp = gsfp;
    if (learn) set_opt(p, *opt);
    const int sub = effective_sub(desc, dgs, gdgs);
    if (desc->rows == 0 || desc->cols == 0) {
        // shared-row gradients of an empty row set are sums over nothing: zero
        if (desc->coef_shared_rows && desc->cols > 0) {
            if (learn) {
                p.nsub = static_cast<uint32_t>(desc->cols / sub);
                return map_cuda(launch_shared_finalize(desc->fmt, sub, p, st));
            }
            cudaError_t e = cudaSuccess;
            if (gcrs) e = cudaMemsetAsync(gcrs, 0, sizeof(float) * (desc->cols / desc->block), st);
            if (e == cudaSuccess && gdgs)
                e = cudaMemsetAsync(gdgs, 0, sizeof(float) * (desc->cols / desc->sub_block), st);
            return map_cuda(e);
        }
        return FOCUS_OK;
    }
    if (!x || !g || (desc->fmt == FOCUS_NVFP4 && !alpha)) return FOCUS_ERR_INVALID_ARG;
    if (!gx && !want_T && !gsfp && !learn) return FOCUS_OK;
    if (desc->coef_shared_rows && want_T) {
        const size_t need = bwd_ws_bytes(desc);
        if (!ws || ws_bytes < need) return FOCUS_ERR_WORKSPACE;
        if (misaligned(ws, 16)) return FOCUS_ERR_MISALIGNED;
        p.ws = static_cast<float*>(ws);
        p.nsub = static_cast<uint32_t>(desc->cols / sub);
        const uint32_t ny = shared_groups(desc);
        return map_cuda(launch_bwd_shared(desc->fmt, desc->dtype, sub, p, ny, st));
    }
    return map_cuda(launch_bwd(desc->fmt, desc->dtype, sub, p, st));
}

size_t bwd_ws_bytes(const focus_desc_t* d)
{
    if (!d->coef_shared_rows || d->rows == 0 || d->cols == 0) return 0;
    const uint32_t ny = shared_groups(d);
    return static_cast<size_t>(ny) * static_cast<size_t>(d->cols / d->sub_block) * 2 * sizeof(float);
}

}  // namespace
}  // namespace focus

using namespace focus;

FOCUS_API int focus_version(void) { return 210; }

FOCUS_API const char* focus_status_string(int status)
{
    switch (status) {
    case FOCUS_OK: return "ok";
    case FOCUS_ERR_INVALID_ARG: return "invalid argument";
    case FOCUS_ERR_UNSUPPORTED: return "unsupported block / sub-block / size";
    case FOCUS_ERR_MISALIGNED: return "misaligned pointer or leading dimension";
    case FOCUS_ERR_WORKSPACE: return "workspace missing or too small";
    case FOCUS_ERR_CUDA: return "CUDA runtime error";
    default: return "unknown status";
    }
}

FOCUS_API size_t focus_workspace_bytes(const focus_desc_t* desc, int which)
{
    if (which == FOCUS_WS_ALPHA) {
        if (check_desc(desc, false) != FOCUS_OK) return 0;
        const uint32_t n = static_cast<uint32_t>(desc->rows * (desc->cols / 8));
        return static_cast<size_t>(alpha_grid(n)) * sizeof(float);
    }
    if (which == FOCUS_WS_BWD) {
        if (check_desc(desc, true) != FOCUS_OK) return 0;
        return bwd_ws_bytes(desc);
    }
    return 0;
}

FOCUS_API int focus_nvfp4_alpha(const focus_desc_t* desc, const void* x, float* alpha_out,
                                void* ws, size_t ws_bytes, focus_stream_t stream)
{
    int rc = check_desc(desc, false);
    if (rc) return rc;
    const bool empty = desc->rows == 0 || desc->cols == 0;
    if (!alpha_out || (!empty && !x)) return FOCUS_ERR_INVALID_ARG;
    if (misaligned(x, 16) || misaligned(alpha_out, 4) || misaligned(ws, 16)) return FOCUS_ERR_MISALIGNED;
    KParams p = make_params(desc);
    const size_t need = static_cast<size_t>(alpha_grid(p.n_chunks)) * sizeof(float);
    if (!empty && (!ws || ws_bytes < need)) return FOCUS_ERR_WORKSPACE;
    p.x = x;
    p.ws = static_cast<float*>(ws);
    return map_cuda(launch_alpha(desc->dtype, p, alpha_out, reinterpret_cast<cudaStream_t>(stream)));
}

FOCUS_API int focus_fq_fwd(const focus_desc_t* desc, const void* x, const float* crs,
                           const float* dgs, const float* alpha, const float* sfp, void* y,
                           uint8_t* scale_bytes, focus_stream_t stream)
{
    int rc = check_desc(desc, true);
    if (rc) return rc;
    if (sfp && desc->coef_shared_rows) return FOCUS_ERR_INVALID_ARG;
    if (desc->rows == 0 || desc->cols == 0) return FOCUS_OK;
    if (!x || !y || (desc->fmt == FOCUS_NVFP4 && !alpha)) return FOCUS_ERR_INVALID_ARG;
    if (rows_misaligned(x, y, nullptr) || misaligned(alpha, 4) || misaligned(sfp, 4))
        return FOCUS_ERR_MISALIGNED;
    if ((rc = check_coef_ptrs(crs, dgs, nullptr, nullptr))) return rc;
    KParams p = make_params(desc);
    p.half = rows_half(desc, x, y, nullptr);
    p.x = x;
    p.y = y;
    p.crs = crs;
    p.dgs = dgs;
    p.alpha = alpha;
    p.sfp = sfp;
    p.scales = scale_bytes;
    return map_cuda(launch_fwd(desc->fmt, desc->dtype, effective_sub(desc, dgs, nullptr), p,
                               reinterpret_cast<cudaStream_t>(stream)));
}

namespace focus {
namespace {

int run_pack(const focus_desc_t* desc, const void* x, const float* crs, const float* dgs,
             const float* alpha, const float* sfp, uint8_t* codes, uint8_t* scale_bytes,
             bool mma_layout, cudaStream_t st)
{
    int rc = check_desc(desc, true);
    if (rc) return rc;
    if (sfp && desc->coef_shared_rows) return FOCUS_ERR_INVALID_ARG;
    if (desc->rows == 0 || desc->cols == 0) return FOCUS_OK;
    if (!x || !codes || !scale_bytes || (desc->fmt == FOCUS_NVFP4 && !alpha))
        return FOCUS_ERR_INVALID_ARG;
    if (rows_misaligned(x, nullptr, nullptr) || misaligned(codes, 16) || misaligned(alpha, 4) ||
        misaligned(sfp, 4))
        return FOCUS_ERR_MISALIGNED;
    if (mma_layout && misaligned(scale_bytes, 16)) return FOCUS_ERR_MISALIGNED;
    if ((rc = check_coef_ptrs(crs, dgs, nullptr, nullptr))) return rc;
    KParams p = make_params(desc);
    p.half = rows_half(desc, x, nullptr, nullptr);
    p.x = x;
    p.crs = crs;
    p.dgs = dgs;
    p.alpha = alpha;
    p.sfp = sfp;
    p.codes = codes;
    p.scales = scale_bytes;
    if (mma_layout) {
        const int64_t sc = desc->cols / desc->block;
        p.sf_tile_cols = static_cast<uint32_t>((sc + 3) / 4);
        // padding of the last tile row / column: zero bytes
        if (desc->rows % 128 != 0 || sc % 4 != 0) {
            const cudaError_t e = cudaMemsetAsync(scale_bytes, 0, mma_scale_bytes(desc), st);
            if (e != cudaSuccess) return FOCUS_ERR_CUDA;
        }
    }
    return map_cuda(launch_pack(desc->fmt, desc->dtype, effective_sub(desc, dgs, nullptr), p, st));
}

}  // namespace
}  // namespace focus

FOCUS_API int focus_pack(const focus_desc_t* desc, const void* x, const float* crs,
                         const float* dgs, const float* alpha, const float* sfp, uint8_t* codes,
                         uint8_t* scale_bytes, focus_stream_t stream)
{
    return run_pack(desc, x, crs, dgs, alpha, sfp, codes, scale_bytes, false,
                    reinterpret_cast<cudaStream_t>(stream));
}

FOCUS_API size_t focus_mma_scale_bytes(const focus_desc_t* desc)
{
    if (check_desc(desc, true) != FOCUS_OK) return 0;
    return mma_scale_bytes(desc);
}

FOCUS_API int focus_pack_mma(const focus_desc_t* desc, const void* x, const float* crs,
                             const float* dgs, const float* alpha, const float* sfp,
                             uint8_t* codes, uint8_t* scale_tiles, focus_stream_t stream)
{
    return run_pack(desc, x, crs, dgs, alpha, sfp, codes, scale_tiles, true,
                    reinterpret_cast<cudaStream_t>(stream));
}

FOCUS_API int focus_fq_bwd(const focus_desc_t* desc, const void* x, const float* crs,
                           const float* dgs, const float* alpha, const float* sfp, const void* g,
                           void* gx, float* gcrs, float* gdgs, float* gsfp, void* ws,
                           size_t ws_bytes, focus_stream_t stream)
{
    return run_bwd(desc, x, crs, dgs, alpha, sfp, g, gx, gcrs, gdgs, gsfp, ws, ws_bytes,
                   reinterpret_cast<cudaStream_t>(stream), nullptr);
}

FOCUS_API int focus_fq_bwd_adamw(const focus_desc_t* desc, const void* x, float* crs, float* dgs,
                                 const float* alpha, float* sfp, const void* g, void* gx,
                                 const focus_adamw_t* hp, const focus_adamw_state_t* state,
                                 const int64_t* step, float* gcrs, float* gdgs, float* gsfp,
                                 void* ws, size_t ws_bytes, focus_stream_t stream)
{
    const OptArgs opt = {crs, dgs, sfp, hp, state, step};
    return run_bwd(desc, x, crs, dgs, alpha, sfp, g, gx, gcrs, gdgs, gsfp, ws, ws_bytes,
                   reinterpret_cast<cudaStream_t>(stream), &opt);
}

// ---------------------------------------------------------------------------
// Group entry points
// ---------------------------------------------------------------------------
namespace focus {
namespace {

enum GroupMode { kGroupAlpha, kGroupFwd, kGroupPack, kGroupBwd };

// Validate a group and fill g (non-empty tensors only); fmt / dt / sub /
// sfpg describe the kernel to run.
int build_group(const focus_tensor_t* t, int n, GroupMode mode, KGroup& g, int& dt, int& fmt, int& sub,
                bool& sfpg)
{
    if (n < 0) return FOCUS_ERR_INVALID_ARG;
    if (n > kMaxGroup) return FOCUS_ERR_UNSUPPORTED;
    if (n > 0 && !t) return FOCUS_ERR_INVALID_ARG;
    std::memset(&g, 0, sizeof(g));
    bool any_dgs = false;
    sfpg = false;
    uint64_t total = 0;
    for (int i = 0; i < n; ++i) {
        const focus_desc_t& d = t[i].desc;
        const focus_tensor_t& a = t[i];
        int rc = check_desc(&d, mode != kGroupAlpha);
        if (rc) return rc;
        const focus_desc_t& d0 = t[0].desc;
        if (d.dtype != d0.dtype) return FOCUS_ERR_INVALID_ARG;
        if (mode != kGroupAlpha) {
            if (d.fmt != d0.fmt || d.block != d0.block || d.sub_block != d0.sub_block || d.ste != d0.ste ||
                d.mx_rule != d0.mx_rule)
                return FOCUS_ERR_INVALID_ARG;
            if (d.coef_shared_rows) return FOCUS_ERR_INVALID_ARG;
            if ((rc = check_coef_ptrs(a.crs, a.dgs, a.gcrs, a.gdgs))) return rc;
            if (misaligned(a.alpha, 4) || misaligned(a.sfp, 4) || misaligned(a.gsfp, 4))
                return FOCUS_ERR_MISALIGNED;
        }
        const bool empty = d.rows == 0 || d.cols == 0;
        if (empty && mode != kGroupAlpha) continue;   // (an empty tensor's alpha is 0)
        if (!empty && !a.x) return FOCUS_ERR_INVALID_ARG;
        if (mode != kGroupAlpha && d.fmt == FOCUS_NVFP4 && !a.alpha) return FOCUS_ERR_INVALID_ARG;
        switch (mode) {
        case kGroupAlpha:
            if (misaligned(a.x, 16)) return FOCUS_ERR_MISALIGNED;
            break;
        case kGroupFwd:
            if (!a.y) return FOCUS_ERR_INVALID_ARG;
            if (rows_misaligned(a.x, a.y, nullptr)) return FOCUS_ERR_MISALIGNED;
            break;
        case kGroupPack:
            if (!a.codes || !a.scale_bytes) return FOCUS_ERR_INVALID_ARG;
            if (rows_misaligned(a.x, nullptr, nullptr) || misaligned(a.codes, 16)) return FOCUS_ERR_MISALIGNED;
            break;
        case kGroupBwd:
            if (!a.g) return FOCUS_ERR_INVALID_ARG;
            if (rows_misaligned(a.x, a.g, a.gx)) return FOCUS_ERR_MISALIGNED;
            if (!a.gx && !a.gcrs && !a.gdgs && !a.gsfp) continue;   // nothing asked of this tensor
            break;
        }
        KParams& p = g.p[g.n];
        p = make_params(&d);
        p.half = mode == kGroupBwd ? rows_half(&d, a.x, a.g, a.gx)
                                   : rows_half(&d, a.x, mode == kGroupFwd ? a.y : nullptr, nullptr);
        p.x = a.x;
        if (mode != kGroupAlpha) {
            p.crs = a.crs;
            p.dgs = a.dgs;
            p.alpha = a.alpha;
            p.sfp = a.sfp;
        }
        if (mode == kGroupFwd) {
            p.y = a.y;
            p.scales = a.scale_bytes;
        } else if (mode == kGroupPack) {
            p.codes = a.codes;
            p.scales = a.scale_bytes;
        } else if (mode == kGroupBwd) {
            p.g = a.g;
            p.gx = a.gx;
            p.gcrs = a.gcrs;
            p.gdgs = a.gdgs;
            p.gsfp = a.gsfp;
            any_dgs |= a.gdgs != nullptr;
            sfpg |= a.sfp != nullptr || a.gsfp != nullptr;
        }
        any_dgs |= a.dgs != nullptr;
        total += mode == kGroupAlpha ? p.n_chunks : p.n_blocks;
        g.n += 1;
    }
    if (total > static_cast<uint64_t>(INT32_MAX)) return FOCUS_ERR_UNSUPPORTED;
    dt = n > 0 ? t[0].desc.dtype : 0;
    fmt = n > 0 ? t[0].desc.fmt : 0;
    sub = (n > 0 && any_dgs) ? t[0].desc.sub_block : (n > 0 ? t[0].desc.block : 16);
    uint32_t at = 0;
    for (int i = 0; i < g.n; ++i) {
        g.start[i] = at;
        at += g.p[i].n_blocks;
    }
    g.start[g.n] = at;
    return FOCUS_OK;
}

// CTAs of the grouped alpha pass: the per-tensor pass's grid for the whole
// group, shared in proportion to the tensors' sizes (at least one each).
void alpha_group_ctas(KGroup& g)
{
    uint64_t total = 0;
    for (int i = 0; i < g.n; ++i) total += g.p[i].n_chunks;
    const uint64_t G = alpha_grid(static_cast<uint32_t>(total));
    uint32_t at = 0;
    for (int i = 0; i < g.n; ++i) {
        g.start[i] = at;
        if (g.p[i].n_chunks > 0)
            at += static_cast<uint32_t>(std::max<uint64_t>(1, G * g.p[i].n_chunks / total));
    }
    g.start[g.n] = at;
}

}  // namespace
}  // namespace focus

FOCUS_API size_t focus_group_workspace_bytes(const focus_tensor_t* t, int n)
{
    KGroup g;
    int dt, fmt, sub;
    bool sfpg;
    if (build_group(t, n, kGroupAlpha, g, dt, fmt, sub, sfpg) != FOCUS_OK) return 0;
    alpha_group_ctas(g);
    return static_cast<size_t>(g.start[g.n]) * sizeof(float);
}

FOCUS_API int focus_nvfp4_alpha_group(const focus_tensor_t* t, int n, float* alpha_out, void* ws,
                                      size_t ws_bytes, focus_stream_t stream)
{
    KGroup g;
    int dt, fmt, sub;
    bool sfpg;
    int rc = build_group(t, n, kGroupAlpha, g, dt, fmt, sub, sfpg);
    if (rc) return rc;
    if (n == 0) return FOCUS_OK;
    if (!alpha_out) return FOCUS_ERR_INVALID_ARG;
    if (misaligned(alpha_out, 4) || misaligned(ws, 16)) return FOCUS_ERR_MISALIGNED;
    alpha_group_ctas(g);
    const size_t need = static_cast<size_t>(g.start[g.n]) * sizeof(float);
    if (need > 0 && (!ws || ws_bytes < need)) return FOCUS_ERR_WORKSPACE;
    g.p[0].ws = static_cast<float*>(ws);
    return map_cuda(launch_alpha_group(dt, g, alpha_out, reinterpret_cast<cudaStream_t>(stream)));
}

FOCUS_API int focus_fq_fwd_group(const focus_tensor_t* t, int n, focus_stream_t stream)
{
    KGroup g;
    int dt, fmt, sub;
    bool sfpg;
    int rc = build_group(t, n, kGroupFwd, g, dt, fmt, sub, sfpg);
    if (rc || g.n == 0) return rc;
    return map_cuda(launch_group_fwd(fmt, dt, sub, g, reinterpret_cast<cudaStream_t>(stream)));
}

FOCUS_API int focus_pack_group(const focus_tensor_t* t, int n, focus_stream_t stream)
{
    KGroup g;
    int dt, fmt, sub;
    bool sfpg;
    int rc = build_group(t, n, kGroupPack, g, dt, fmt, sub, sfpg);
    if (rc || g.n == 0) return rc;
    return map_cuda(launch_group_pack(fmt, dt, sub, g, reinterpret_cast<cudaStream_t>(stream)));
}

FOCUS_API int focus_fq_bwd_group(const focus_tensor_t* t, int n, focus_stream_t stream)
{
    KGroup g;
    int dt, fmt, sub;
    bool sfpg;
    int rc = build_group(t, n, kGroupBwd, g, dt, fmt, sub, sfpg);
    if (rc || g.n == 0) return rc;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    return map_cuda(fmt == 0 ? launch_group_bwd_mx(dt, sub, sfpg, g, st) : launch_group_bwd_nv(dt, sub, sfpg, g, st));
}
