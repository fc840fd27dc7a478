/*
 * focus_fq.h -- C ABI of the FOCUS FP4 fake-quantizer for GB300 (sm_103a).
 *
 * FOCUS (Coupled-Relaxation and Dual-Granularity Scaling) learns the FP4
 * quantization scale S^q separately from the stored, hardware-format
 * dequantization scale S^dq.  Per block i of B contiguous elements along a
 * row (B = 32 for MXFP4, 16 for NVFP4) and per sub-block k of b elements:
 *
 *   m_i      = max |x| over block i                              (Eq. 2-3)
 *   S^dq_i   = MXFP4: 2^e_i, e_i from the E8M0 rule               (Eq. 3)
 *              NVFP4: alpha * Q_E4M3(m_i / (alpha * 6))           (Eq. 2)
 *   S^q_ik   = S^dq_i * c_i * c_i^k                               (Eq. 6, Eq. 8)
 *   xbar     = Q_E2M1(x / S^q_ik),  y = xbar * S^dq_i             (Eq. 1, 7, 8)
 *
 * c_i is the per-block CRS coefficient (Sec. 3.3), c_i^k the per-sub-block
 * DGS coefficient (Sec. 3.4).  The backward pass is the straight-through
 * estimator the paper applies to every non-differentiable operation
 * (Sec. 3.2).  The export writes what the deployed model keeps: FP4 codes and
 * the dequantization scales (Fig. 3(d)).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All tensor pointers are DEVICE pointers owned by the caller.  The library
 *   allocates nothing, keeps no pointer after a call returns and never
 *   synchronises the host: work is enqueued on `stream` (NULL = the legacy
 *   default stream) and completes asynchronously.
 * - x, y, g and gx are row-major [rows, ld] arrays of desc->dtype; only the
 *   first `cols` elements of each row are read or written.  Every row must
 *   start on a 16-byte boundary: the arrays 16-byte aligned and
 *   ld * sizeof(element) a multiple of 16 (FOCUS_ERR_MISALIGNED otherwise).
 *   When every row of every array of a call starts on a 32-byte boundary
 *   (arrays 32-byte aligned, ld * sizeof(element) a multiple of 32) the
 *   kernels move each 32-byte piece of a row with one 256-bit access, else
 *   with two 128-bit accesses; the results are the same.
 * - Coefficient arrays are dense fp32: crs / gcrs are [rows, cols/block] and
 *   dgs / gdgs are [rows, cols/sub_block]; with coef_shared_rows = 1 both are
 *   a single row ([cols/block], [cols/sub_block]) shared by all rows.  They
 *   must be 16-byte aligned.  A NULL crs or dgs means "all coefficients 1".
 * - Scale bytes are dense uint8 [rows, cols/block] (E8M0 biased exponent for
 *   MXFP4, E4M3FN for NVFP4).  Codes are dense uint8 [rows, cols/2]: element
 *   2t of a row in the low nibble of byte t, element 2t+1 in the high nibble;
 *   a code is sign(1) | E2M1 magnitude index(3).  Codes must be 16-byte aligned.
 * - Every call returns FOCUS_OK (0) or a negative focus_status_t.  Argument
 *   errors are detected on the host before anything is launched; a launch
 *   failure is reported as FOCUS_ERR_CUDA (cudaGetLastError is consumed).
 * - Preconditions that are documented but not checked on the hot path: x and
 *   g finite; coefficients finite and > 0; alpha finite and >= 0.  A
 *   sub-block whose S^dq or S^q is zero or infinite is "dead": it yields
 *   codes 0, values +0, input gradient +0 and no coefficient gradient.
 * - Results are deterministic: no atomics, fixed reduction orders.
 */
#ifndef FOCUS_FQ_H
#define FOCUS_FQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Opaque CUDA stream handle; identical to cudaStream_t. */
typedef struct CUstream_st* focus_stream_t;

typedef enum {
    FOCUS_OK = 0,
    FOCUS_ERR_INVALID_ARG = -1,   /* NULL where required, bad enum, ld < cols, ... */
    FOCUS_ERR_UNSUPPORTED = -2,   /* block / sub-block / size outside what is built */
    FOCUS_ERR_MISALIGNED = -3,    /* pointer or ld alignment rule broken */
    FOCUS_ERR_WORKSPACE = -4,     /* workspace NULL or smaller than required */
    FOCUS_ERR_CUDA = -5           /* the CUDA runtime reported an error */
} focus_status_t;

typedef enum { FOCUS_MXFP4 = 0, FOCUS_NVFP4 = 1 } focus_format_t;
typedef enum { FOCUS_F32 = 0, FOCUS_BF16 = 1, FOCUS_F16 = 2 } focus_dtype_t;
typedef enum { FOCUS_STE_IDENTITY = 0, FOCUS_STE_CLIPPED = 1 } focus_ste_t;
typedef enum { FOCUS_MX_CEIL = 0, FOCUS_MX_FLOOR = 1 } focus_mx_rule_t;

/* Tensor and method descriptor (host memory, read during the call only).
 *   rows, cols, ld    x is [rows, ld] row-major, blocks run along cols;
 *                     cols % block == 0; rows * cols / 8 < 2^31.
 *   dtype             focus_dtype_t of x, y, g and gx (binary32, bfloat16 or
 *                     IEEE binary16; 16-bit outputs are rounded to nearest
 *                     even, binary16 overflowing to infinity).
 *   fmt               focus_format_t.
 *   block             32 for FOCUS_MXFP4, 16 for FOCUS_NVFP4 (Sec. 3.1).
 *   sub_block         DGS sub-block size b (Sec. 3.4): one of 2, 4, 8, 16,
 *                     32 dividing block; b == block means K = 1 (CRS only).
 *                     The paper uses 8 for both formats.
 *   coef_shared_rows  0: coefficients per (row, block); 1: one set shared by
 *                     all rows (channel-block coefficients of activations).
 *   ste               focus_ste_t: IDENTITY passes the gradient through
 *                     Q_E2M1 unchanged; CLIPPED zeroes it where |x/S^q| > 6.
 *   mx_rule           focus_mx_rule_t, MXFP4 only: CEIL e = ceil(log2(m/6))
 *                     (the paper's "typically ceiling", Eq. 3), or the OCP
 *                     MX v1.0 rule e = floor(log2 m) - 2. */
typedef struct {
    int64_t rows;
    int64_t cols;
    int64_t ld;
    int32_t dtype;
    int32_t fmt;
    int32_t block;
    int32_t sub_block;
    int32_t coef_shared_rows;
    int32_t ste;
    int32_t mx_rule;
} focus_desc_t;

/* Which workspace focus_workspace_bytes reports. */
enum { FOCUS_WS_ALPHA = 0, FOCUS_WS_BWD = 1 };

/* NVFP4 per-tensor scale, Eq. 2: alpha = max|x| / (M_FP4 * M_FP8)
 * = fl(max|x| / 2688), written as one fp32 to *alpha_out (device).
 * For weights the paper computes alpha once and freezes it (Sec. 3.2); for
 * dynamically quantized activations it is recomputed on every call.
 * ws: device scratch of at least focus_workspace_bytes(desc, FOCUS_WS_ALPHA)
 * bytes, 16-byte aligned; its contents are overwritten.  desc->fmt, block and
 * sub_block are not used. */
int focus_nvfp4_alpha(const focus_desc_t* desc, const void* x, float* alpha_out,
                      void* ws, size_t ws_bytes, focus_stream_t stream);

/* focus_nvfp4_alpha for callers that cannot allocate device memory.  The
 * paper has no counterpart: this is a deployment aid of this library.
 * Computes exactly what focus_nvfp4_alpha computes, but takes no workspace:
 * the per-CTA partial maxima live in a 16 KiB array inside the library's own
 * device memory (4096 fp32 slots, held by every GPU that loads the library
 * until the process exits).  Meant for code that is handed only its input
 * and output buffers -- e.g. a plugin inside a host application that owns
 * every device allocation -- or that must never call cudaMalloc on its hot
 * path because that call can synchronise the device.  It calls no
 * allocating routine.
 * - The first call on a device looks up the array's device address (with
 *   that device current) and caches it for the life of the process; make
 *   that first call before any stream capture.  The cached address belongs
 *   to the device's current context: after cudaDeviceReset (or anything else
 *   that destroys the primary context) this entry point must not be called
 *   again in the same process.
 * - Every call on a device shares the one array, so calls that overlap on
 *   the GPU (e.g. on two streams at once) race and may return wrong values;
 *   serialise them.  Nothing in the array needs clearing between calls.
 * - Returns FOCUS_ERR_WORKSPACE if the pass would need more than 4096
 *   partial slots (a GPU with more than 512 SMs). */
int focus_nvfp4_alpha_noalloc(const focus_desc_t* desc, const void* x, float* alpha_out,
                              focus_stream_t stream);

/* Fake-quantization forward, Eq. 1-3 and 6-8: y = Q_E2M1(x / S^q) * S^dq.
 * x      [rows, ld] input (read only).
 * crs    CRS coefficients c_i, or NULL for 1 (Eq. 6-7).
 * dgs    DGS coefficients c_i^k, or NULL for 1 (Eq. 8).
 * alpha  NVFP4: device pointer to the fp32 per-tensor scale (required);
 *        MXFP4: ignored (may be NULL).
 * sfp    optional learnable full-precision scales S^fp, dense fp32
 *        [rows, cols/block], finite and >= 0 (Eq. 4): S^dq = Q_fmt(S^fp)
 *        replaces the absmax scale -- MXFP4: the ceiling power of two of
 *        S^fp (mx_rule is not used); NVFP4: S^fp is the learnable Delta,
 *        S^dq = alpha * Q_E4M3(S^fp) with alpha frozen.  NULL: the absmax
 *        scale of Eq. 2-3.  Not with coef_shared_rows = 1 (INVALID_ARG).
 * y      [rows, ld] output in dtype (may alias nothing else).
 * scale_bytes  optional [rows, cols/block] output of the stored scale bytes. */
int focus_fq_fwd(const focus_desc_t* desc, const void* x, const float* crs,
                 const float* dgs, const float* alpha, const float* sfp, void* y,
                 uint8_t* scale_bytes, focus_stream_t stream);

/* Straight-through-estimator backward (Sec. 3.2) of focus_fq_fwd.
 * x, crs, dgs, alpha, sfp  as for focus_fq_fwd.
 * g      [rows, ld] upstream gradient dL/dy (dtype).
 * gx     optional [rows, ld] output dL/dx = mask * fl(g * fl(S^dq / S^q)), the
 *        scale ratio rounded once per sub-block; NULL skips it (frozen
 *        weights, Sec. 3.2).
 * gcrs   optional dL/dc_i    = -sum_k T_ik * c_i^k / (c_i c_i^k)^2
 * gdgs   optional dL/dc_i^k  = -T_ik * c_i / (c_i c_i^k)^2
 *        with T_ik = sum over sub-block (i,k) of mask * g * x; in shared mode
 *        both are also summed over rows.  They are written (not accumulated).
 *        Requesting gcrs with crs == NULL gives the gradient at c_i = 1
 *        (likewise gdgs with dgs == NULL).
 * gsfp   optional [rows, cols/block] output dL/dS^fp (Eq. 4 with the STE
 *        through Q_fmt): dL/dS^dq_i = sum over block i of
 *        g * (q - mask * x / S^q) (q the E2M1 value, S^q = S^dq c_i c_i^k
 *        taken exactly), times alpha for NVFP4.  With sfp == NULL it is the
 *        gradient at the absmax initialisation.  Per-row coefficients only.
 * ws     device scratch of focus_workspace_bytes(desc, FOCUS_WS_BWD) bytes
 *        (zero when coef_shared_rows == 0, in which case ws may be NULL).
 * Coefficient gradients are computed with compensated (double-fp32)
 * arithmetic and match an exact evaluation to about 1e-5 relative. */
int focus_fq_bwd(const focus_desc_t* desc, const void* x, const float* crs,
                 const float* dgs, const float* alpha, const float* sfp, const void* g,
                 void* gx, float* gcrs, float* gdgs, float* gsfp, void* ws, size_t ws_bytes,
                 focus_stream_t stream);

/* AdamW hyper-parameters (host memory, read during the call).  The paper
 * trains with AdamW at a constant learning rate, one rate for the block
 * scale S^fp and one for the relaxation coefficients (Sec. 4.1: MXFP4
 * 2e-2 / 5e-2, NVFP4 5e-3 / 1e-3).  Requirements: learning rates and
 * weight_decay finite and >= 0, 0 <= beta1, beta2 < 1, eps finite and > 0;
 * otherwise FOCUS_ERR_INVALID_ARG. */
typedef struct {
    float lr_coef;        /* learning rate of c_i and c_i^k */
    float lr_scale;       /* learning rate of S^fp */
    float beta1;          /* first-moment decay (PyTorch default 0.9) */
    float beta2;          /* second-moment decay (PyTorch default 0.999) */
    float eps;            /* denominator guard (PyTorch default 1e-8) */
    float weight_decay;   /* decoupled decay lambda (PyTorch AdamW default 0.01) */
} focus_adamw_t;

/* Optimizer state: fp32 moment arrays shaped and laid out exactly like the
 * parameter they belong to (16-byte aligned, caller-owned device memory,
 * zero before the first step).  Pairs of a parameter that is not learned
 * (NULL in focus_fq_bwd_adamw) are ignored. */
typedef struct {
    float* m_crs;
    float* v_crs;
    float* m_dgs;
    float* v_dgs;
    float* m_sfp;
    float* v_sfp;
} focus_adamw_state_t;

/* STE backward fused with one AdamW step on the learnable arrays (Sec. 3.2
 * and Sec. 4.1).  Computes exactly what focus_fq_bwd computes, at the
 * parameter values on entry, then, for each of crs, dgs and sfp that is
 * non-NULL (the arrays being learned), replaces it in place by
 *   p <- p * (1 - lr * weight_decay)
 *   m <- beta1 * m + (1 - beta1) * grad,  v <- beta2 * v + (1 - beta2) * grad^2
 *   p <- p - lr / (1 - beta1^t) * m / (sqrt(v) / sqrt(1 - beta2^t) + eps)
 * (PyTorch's AdamW) with lr = hp->lr_scale for sfp and hp->lr_coef for the
 * coefficients, in binary32, and writes the new moments.  The moments are
 * correctly rounded binary32 operations; the square root and the division of
 * the last line are the hardware's approximate forms (within 2 ulp each), so
 * the new parameters may differ from a correctly rounded evaluation by a few
 * ulp.  The gradients are not written to memory unless gcrs / gdgs / gsfp
 * are given.
 * crs, dgs, sfp  parameters as for focus_fq_bwd, updated in place; NULL: not
 *        learned (coefficient 1 / absmax scale).  sfp only with per-row
 *        coefficients.
 * step   device pointer to an int64 t >= 1, the number of this update (the
 *        caller advances it before each step; the library only reads it, so
 *        a captured CUDA graph that advances it replays correctly).
 * With coef_shared_rows = 1 the step is applied once the gradient summed
 * over all rows is complete (an empty row set gives gradient 0, and the
 * step still applies).  Other arguments as for focus_fq_bwd. */
int focus_fq_bwd_adamw(const focus_desc_t* desc, const void* x, float* crs, float* dgs,
                       const float* alpha, float* sfp, const void* g, void* gx,
                       const focus_adamw_t* hp, const focus_adamw_state_t* state,
                       const int64_t* step, float* gcrs, float* gdgs, float* gsfp, void* ws,
                       size_t ws_bytes, focus_stream_t stream);

/* Export (Fig. 3(d)): the FP4 codes of Q_E2M1(x / S^q) and the scale bytes
 * of S^dq -- what the deployed MXFP4 / NVFP4 model stores; S^q and the
 * coefficients are not part of it.  NVFP4 also needs the caller's alpha.
 * x, crs, dgs, alpha, sfp  as for focus_fq_fwd.
 * codes        [rows, cols/2] uint8 output (required).
 * scale_bytes  [rows, cols/block] uint8 output (required). */
int focus_pack(const focus_desc_t* desc, const void* x, const float* crs,
               const float* dgs, const float* alpha, const float* sfp, uint8_t* codes,
               uint8_t* scale_bytes, focus_stream_t stream);

/* Export for the Blackwell block-scaled tensor-core MMA (the deployment the
 * paper targets: FP4 GEMMs on hardware that reads E2M1 codes with E8M0 /
 * E4M3 block scales directly, Sec. 1 and Sec. 3.1).  Codes exactly as
 * focus_pack writes them (row-major, K-major operand of the MMA).  The scale
 * bytes go to scale_tiles in the MMA scale-factor layout: the [rows, C]
 * scale matrix (C = cols / block) is cut into tiles of 128 rows x 4 columns
 * of 512 bytes; tile (i, j) starts at byte (i * ceil(C / 4) + j) * 512, and
 * inside it row r (0..127) and column c (0..3) are at byte
 * (r % 32) * 16 + (r / 32) * 4 + c.  Bytes of the padding (rows beyond
 * `rows`, columns beyond C) are written as 0.  scale_tiles: 16-byte aligned,
 * focus_mma_scale_bytes(desc) bytes.  Other arguments as for focus_pack. */
int focus_pack_mma(const focus_desc_t* desc, const void* x, const float* crs,
                   const float* dgs, const float* alpha, const float* sfp, uint8_t* codes,
                   uint8_t* scale_tiles, focus_stream_t stream);

/* Size in bytes of focus_pack_mma's scale tiles for this descriptor
 * (ceil(rows / 128) * ceil(cols / block / 4) * 512); 0 for an invalid
 * descriptor. */
size_t focus_mma_scale_bytes(const focus_desc_t* desc);

/* W4A4 GEMM on the block-scaled FP4 tensor cores (tcgen05.mma
 * .kind::mxf4 / .kind::mxf4nvf4) over two focus_pack_mma exports, the
 * product a deployed FOCUS model computes with nothing but its export
 * (Sec. 1, Sec. 3.1; Fig. 3(d)):
 *   D[m, n] = sum_k A[m, k] * B[n, k]                       (MXFP4)
 *   D[m, n] = fl(alpha_a * alpha_b) * sum_k A[m, k] * B[n, k]  (NVFP4)
 * with A[m, k] = E2M1(code) * scale(m, k / block) (E8M0 / E4M3 scales).
 * a_codes [M, K/2], b_codes [N, K/2]: row-major code bytes as written by
 * focus_pack_mma (B is the second operand's rows, e.g. a weight [out, in]);
 * a_scale_tiles / b_scale_tiles: their MMA-layout scale tiles; alpha_a,
 * alpha_b: device fp32 per-tensor scales (NVFP4 only; ignored for MXFP4).
 * d: [M, ldd] row-major output (ldd >= N) of d_dtype (FOCUS_F32, or
 * FOCUS_BF16 rounded to nearest even), overwritten.  The products are exact
 * and accumulate in fp32 inside the tensor core; alpha is applied to the
 * fp32 sum before the output rounding.
 * Requirements: K % 32 == 0 (FOCUS_ERR_UNSUPPORTED otherwise: code rows on
 * 16-byte boundaries); codes and
 * scale tiles 16-byte aligned.  timeout_flag: optional device int32; a
 * kernel whose wait on its pipeline gives up sets it to 1 (the output is
 * then incomplete) instead of waiting for ever.  Enqueued on `stream`; the
 * kernel is persistent and launched in clusters of two CTAs (one per SM),
 * each pair computing 256 x 256 tiles of D with the tensor cores of both of
 * its SMs; every CTA loads its own operand tiles. */
int focus_fp4_gemm(int32_t fmt, int64_t M, int64_t N, int64_t K, const uint8_t* a_codes,
                   const uint8_t* a_scale_tiles, const float* alpha_a, const uint8_t* b_codes,
                   const uint8_t* b_scale_tiles, const float* alpha_b, void* d, int32_t d_dtype,
                   int64_t ldd, int32_t* timeout_flag, focus_stream_t stream);

/* ---- Group entry points --------------------------------------------------
 * One launch for several tensors, e.g. all projections of a transformer
 * layer: the kernel walks the blocks of all tensors as one range, so no
 * tensor's tail runs alone on a mostly idle GPU and per-tensor launches are
 * saved.  Every result is exactly the per-tensor entry point's, bit for bit
 * (each block is computed by the same code from the same inputs).
 *
 * Each tensor is described by one focus_tensor_t (host memory, read during
 * the call); the fields a call does not use are ignored.  Rules, checked on
 * the host before anything is launched:
 * - 0 <= n <= FOCUS_MAX_GROUP (FOCUS_ERR_UNSUPPORTED above);
 * - all descriptors share fmt, dtype, block, sub_block, ste and mx_rule
 *   (FOCUS_ERR_INVALID_ARG otherwise); coef_shared_rows must be 0 (shared
 *   coefficients: use the per-tensor entry points);
 * - each tensor obeys the per-tensor entry point's rules (pointers,
 *   alignment, required outputs); empty tensors are skipped;
 * - at most 2^31 - 1 blocks in total. */
#define FOCUS_MAX_GROUP 16

typedef struct {
    focus_desc_t desc;
    const void* x;          /* input                                  (all)  */
    const void* g;          /* upstream gradient dL/dy                (bwd)  */
    void* y;                /* fake-quantized output                  (fwd)  */
    void* gx;               /* optional dL/dx                         (bwd)  */
    const float* crs;       /* optional c_i                                  */
    const float* dgs;       /* optional c_i^k                                */
    const float* alpha;     /* NVFP4 per-tensor scale (device; fwd, bwd, pack) */
    const float* sfp;       /* optional learnable S^fp                       */
    float* gcrs;            /* optional dL/dc_i                       (bwd)  */
    float* gdgs;            /* optional dL/dc_i^k                     (bwd)  */
    float* gsfp;            /* optional dL/dS^fp                      (bwd)  */
    uint8_t* codes;         /* export codes                           (pack) */
    uint8_t* scale_bytes;   /* scale bytes: optional (fwd), required (pack) */
} focus_tensor_t;

/* focus_nvfp4_alpha for each tensor (Eq. 2); alpha_out: n device floats.
 * ws: focus_group_workspace_bytes(t, n) bytes of device scratch, 16-byte
 * aligned.  desc->fmt / sub_block are not used. */
int focus_nvfp4_alpha_group(const focus_tensor_t* t, int n, float* alpha_out, void* ws,
                            size_t ws_bytes, focus_stream_t stream);
/* Scratch that focus_nvfp4_alpha_group needs for these tensors (0 if the
 * group is invalid). */
size_t focus_group_workspace_bytes(const focus_tensor_t* t, int n);
/* focus_fq_fwd for each tensor (Eq. 1-8). */
int focus_fq_fwd_group(const focus_tensor_t* t, int n, focus_stream_t stream);
/* focus_fq_bwd for each tensor (Sec. 3.2), per-row coefficients only. */
int focus_fq_bwd_group(const focus_tensor_t* t, int n, focus_stream_t stream);
/* focus_pack for each tensor (Fig. 3(d)), row-major scale bytes. */
int focus_pack_group(const focus_tensor_t* t, int n, focus_stream_t stream);

/* Device scratch (bytes) that focus_nvfp4_alpha (which = FOCUS_WS_ALPHA) or
 * focus_fq_bwd (which = FOCUS_WS_BWD) needs for this descriptor on the
 * current device; 0 for an invalid descriptor. */
size_t focus_workspace_bytes(const focus_desc_t* desc, int which);

/* Static, NUL-terminated description of a status code. */
const char* focus_status_string(int status);

/* ABI version of this library (major * 100 + minor): 210. */
int focus_version(void);

#ifdef __cplusplus
}
#endif

#endif /* FOCUS_FQ_H */
