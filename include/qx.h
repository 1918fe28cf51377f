/*
 * qx.h -- C ABI of the GB300 (sm_103a) library for per-group 3/4-bit weight
 * quantization fused into matrix multiplication.
 *
 * The method: a weight matrix W [n][k] (fp16, row n = output feature) is split
 * into groups of g consecutive weights along k, and every group is coded with
 * 3 or 4 bits per weight, either uniformly (equally spaced points, per-group fp16
 * scale and zero-point; paper Section 2.2 and Section 3.2, Q4_0 / Q4_K) or
 * non-uniformly (a per-group codebook, a LUT of 2^b fp16 levels placed where the
 * weights' probability mass is, fit by Lloyd-Max; Section 2.2, Fig. 2a).  The
 * recipe (bits, group size, uniform vs non-uniform) is chosen per matrix
 * (Sections 2.1 and 2.3: per-layer and per-sub-model choices).  Inference
 * dequantizes inside the matrix multiply: decode is memory-bound, so the
 * packing and the unpacking kernels decide its run time (Section 2.4); prefill
 * is a dense contraction (Table 2, "Prefill").
 *
 * Conventions for every entry point
 *   - Buffers are caller-owned.  "device" pointers are CUDA global memory of the
 *     current device; "host" pointers are CPU memory.  The library reads no
 *     buffer after a call's work has run; the decode calls keep their recent
 *     launch plans keyed by the buffer addresses and shapes, and reuse a plan
 *     only when a later call passes the same addresses and shapes again.
 *   - `stream` is a cudaStream_t passed as void*; NULL means the legacy default
 *     stream.  Device work is asynchronous on that stream.
 *   - Arguments are validated on the host before anything is launched; on a
 *     validation failure nothing is launched and a non-zero qx_status returns.
 *   - Errors the device can only detect while running (non-finite weights, a
 *     bounded wait that gave up) set a per-device status word that
 *     qx_get_device_status() reads and clears.
 *   - fp16 values are IEEE binary16 stored as uint16_t; bf16 is not used.
 *
 * Packed layout (the paper prints none; this library fixes it).  k must be a
 * multiple of 128 and of g; rows are stored one after another.
 *   codes, 4-bit : k/2 bytes per row.  Little-endian 32-bit word t holds the
 *                  codes of k = 8t..8t+7; the code of k = 8t+j sits in nibble
 *                  j/2 + 4*(j%2).
 *   codes, 3-bit : 3k/8 bytes per row, three planes of k/8 bytes.  Superblock s
 *                  (k = 128s..128s+127) owns bytes 16s..16s+15 of each plane;
 *                  word i (bytes 4i..4i+3 of those 16) of planes 0/1/2, called
 *                  A_i/B_i/C_i, code k = 128s+32i+m (m = 0..31): bits 0-2 of
 *                  nibble t (t = 0..7) of A_i, B_i, C_i hold the codes of
 *                  m = t, 8+t, 16+t; bit 3 of nibble t of A_i, B_i, C_i holds
 *                  bit 0, 1, 2 of the code of m = 24+t.
 *   scales       : fp16 [n][k/g]                    (uniform only)
 *   zeros        : uint8 [n][ceil(k/g/2)], group j in the low nibble of byte
 *                  j/2 when j is even, else the high nibble (uniform only)
 *   luts         : fp16 [n][k/g][2^bits], ascending (non-uniform only)
 *
 * Dequantized weight (bit-exact contract shared with the CPU oracle):
 *   uniform: w_hat = fp16_rn((float)(q - z) * (float)s)
 *   LUT    : w_hat = luts[n][group][q]
 */
#ifndef QX_H
#define QX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum qx_status {
    QX_OK = 0,
    QX_ERR_INVALID_ARG = 1,  /* NULL pointer, non-positive size, bad enum value   */
    QX_ERR_UNSUPPORTED = 2,  /* well-formed but not built: bits/group/kind/batch   */
    QX_ERR_ALIGNMENT = 3,    /* a pointer breaks the alignment stated below       */
    QX_ERR_CUDA = 4,         /* a CUDA runtime call or a kernel launch failed     */
    QX_ERR_TIMEOUT = 5,      /* device: a bounded wait gave up (device status)    */
    QX_ERR_NONFINITE = 6     /* device: qx_quantize met NaN or Inf (device status) */
} qx_status;

typedef enum qx_kind {
    QX_UNIFORM = 0, /* per-group fp16 scale + 4-bit zero-point, RTN (Section 3.2)   */
    QX_LUT = 1,     /* per-group 2^bits-entry fp16 codebook, Lloyd-Max (Section 2.2) */
    QX_Q4X = 2      /* shared codebooks (Section 3.2): a qx_select_recipe candidate
                       only; every qx_packed entry point rejects it (INVALID_ARG) */
} qx_kind;

typedef enum qx_dtype { QX_F16 = 0, QX_F32 = 1 } qx_dtype;

/* Per-matrix recipe (Sections 2.1-2.3).  Built: uniform bits 3/4 with
 * group_size 32/64/128/256; LUT bits 3 with group_size 32/64/128/256.
 * lloyd_iters (LUT only): Lloyd-Max iteration limit, 0..1000. */
typedef struct qx_recipe {
    int32_t bits;
    int32_t group_size;
    int32_t kind;        /* qx_kind */
    int32_t lloyd_iters;
} qx_recipe;

/* Byte sizes of the packed buffers; 0 for a buffer the recipe does not use. */
typedef struct qx_sizes {
    uint64_t codes, scales, zeros, luts;
} qx_sizes;

/* A packed matrix.  All four pointers are device memory, 16-byte aligned
 * (unused ones may be NULL). */
typedef struct qx_packed {
    int64_t n, k;
    qx_recipe recipe;
    void *codes;
    void *scales;
    void *zeros;
    void *luts;
} qx_packed;

/* Host only: byte sizes of the packed buffers of an n x k matrix, from the
 * packed layout above (the paper gives none: Section 2.4 names the packing
 * kernels and the data-mover bus widths that shape it; this library's reading
 * of them is the layout in the header comment).  The bits per weight of
 * Tables 1-2 are 8 x (these sizes summed) / (n k).
 * Errors: INVALID_ARG (NULL, n < 1, k < 1), UNSUPPORTED (recipe not built or
 * k not a multiple of 128 and of g). */
qx_status qx_packed_size(int64_t n, int64_t k, const qx_recipe *recipe, qx_sizes *out);

/* Quantize and pack W (device fp16 [n][k], row-major, 16-byte aligned) into
 * the caller-allocated buffers of *out (out->n, out->k, out->recipe must equal
 * n, k, *recipe).  Uniform: Section 2.2 / 3.2 RTN with per-group scale and
 * zero-point.  LUT: per-group Lloyd-Max codebook (Section 2.2, Fig. 2a).  Codes,
 * scales, zeros and LUTs are bit-identical to the CPU oracle's.  A non-finite
 * weight sets QX_ERR_NONFINITE in the device status; its group's output is
 * unspecified. */
qx_status qx_quantize(const void *W, int64_t n, int64_t k, const qx_recipe *recipe,
                      const qx_packed *out, void *stream);

/* Dequantize a packed matrix into W_out (device fp16 [n][k], 16-byte aligned),
 * bit-exact with the formula in the header comment (Section 2.4 unpacking). */
qx_status qx_dequant(const qx_packed *p, void *W_out, void *stream);

/* Decode matmul y = x W_hat^T (Section 2.4: memory-bound decoding; Table 2
 * "Decode").  x: device fp16 [batch][k], row-major, 16-byte aligned;
 * y: device [batch][n] of y_dtype (QX_F16 or QX_F32), 4-byte aligned.
 * batch in 1..16; k <= 32768.  The weights are dequantized in registers
 * (w_hat exactly as qx_dequant) and multiplied on the tensor cores with x:
 * the fp16 products are exact and summed in fp32.  One launch streams the
 * weights once for the whole batch. */
qx_status qx_gemv(const qx_packed *p, const void *x, int32_t batch, void *y,
                  int32_t y_dtype, void *stream);

/* Flags of qx_gemv_multi. */
enum {
    /* Launch with programmatic dependent launch: the kernel may start, and
     * stream this call's weights, while the previous kernel in the stream is
     * still running; it waits for that kernel before reading x or writing y.
     * Set it only when the previous kernel does not write this call's weights. */
    QX_GEMV_PDL = 1,
    /* qx_gemv_fused and qx_decode_step_fused only: launch each group on its
     * own (one launch after another on the stream, with QX_GEMV_PDL as given)
     * instead of all groups in one launch; each launch still balances its
     * CTAs with the workspace. */
    QX_GEMV_SEPARATE = 2
};

/* Several decode matmuls in one launch: y[i] = x[i] W_hat_i^T, i < count
 * (count 1..8).  All matrices share bits and kind (the recipe's group size and
 * the shapes may differ); x[i], y[i] are device pointers with the layout and
 * alignment of qx_gemv, passed in host arrays of `count` pointers.  One
 * persistent grid covers the rows of all matrices in byte-balanced slices, so
 * the launch and HBM ramp-up are paid once for the whole group (e.g. the q, k,
 * v or gate, up projections of a decoder layer, which share x).
 * flags: 0 or QX_GEMV_PDL. */
qx_status qx_gemv_multi(const qx_packed *mats, int32_t count, const void *const *x, int32_t batch,
                        void *const *y, int32_t y_dtype, int32_t flags, void *stream);

/* One group of a qx_gemv_chain call: the arguments of one qx_gemv_multi. */
typedef struct qx_gemv_group {
    const qx_packed *mats;   /* count matrices sharing bits and kind */
    int32_t count;           /* 1..8 */
    const void *const *x;    /* count device pointers, as in qx_gemv_multi */
    void *const *y;          /* count device pointers */
} qx_gemv_group;

/* A decode step in one call: qx_gemv_multi(groups[i]...) for i = 0..ngroups-1
 * (ngroups 1..64) in order on `stream`, all with the same batch, y_dtype and
 * flags (e.g. the q,k,v | o | gate,up | down groups of a decoder layer, with
 * QX_GEMV_PDL).  The results equal the separate calls bit for bit; the host
 * cost of the step is one call.  All groups are validated before the first
 * launch; a failing group returns its status and nothing is launched. */
qx_status qx_gemv_chain(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype,
                        int32_t flags, void *stream);

/* A copy of a decode step: `bytes` from src to dst (host to device for the
 * inputs, device to host for the outputs). */
typedef struct qx_copy {
    void *dst;
    const void *src;
    size_t bytes;
} qx_copy;

/* A whole decode step in one call, in order on `stream`: the nin copies `in`
 * (host to device; pinned host memory keeps them asynchronous), the groups as
 * in qx_gemv_chain, the nout copies `out` (device to host), then, when sync is
 * non-zero, a synchronization of the stream (the outputs are then in host
 * memory).  nin, nout 0..16.  Every group is validated before the first copy;
 * a failing argument returns its status and nothing is issued.
 * When every host buffer of a direction is pinned (mapped into the device's
 * address space), every device buffer is device memory and they total at
 * most 4 MiB, that direction's copies are made by one small kernel of the
 * library that reads or writes the host buffers through their device
 * addresses (the copy out starts early under programmatic dependent launch
 * and waits in the kernel for the groups to finish); otherwise by
 * cudaMemcpyAsync, one per buffer.  Either way the bytes are the same.
 * When every host buffer is pinned and `stream` is not being captured, the
 * first call with a given set of arguments captures the copies and launches
 * as a CUDA graph (on a stream of the library's own) and every later call
 * with the same arguments replays it: one launch per step.  The library keeps
 * up to 16 such graphs, and the device memory they hold, until the process
 * ends.  Otherwise the copies and launches are issued one by one. */
qx_status qx_decode_step(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups,
                         int32_t batch, int32_t y_dtype, int32_t flags, const qx_copy *out, int32_t nout,
                         int32_t sync, void *stream);

/* Bytes of workspace qx_gemv_fused and qx_decode_step_fused need (host only;
 * a constant, about 1 MiB). */
qx_status qx_gemv_fused_workspace(size_t *bytes);

/* The groups of qx_gemv_chain (Section 2.4: decoding is memory-bound, so the
 * weight stream should not stop between the projections of a layer) in ONE
 * persistent launch: one CTA per SM streams the weights of every group without
 * a break, and group i + 1 reads its x only once every CTA has finished group
 * i (its y written), so x of a later group may be the y of an earlier one.
 * ngroups 1..64; the groups run as one launch when there are at most 4 of them
 * with at most 16 matrices in all, sharing bits and kind, and flags do not ask
 * for QX_GEMV_SEPARATE (else one launch per group, one after another).
 * Every launch splits its work between the CTAs at 1024-weight slices of a
 * 32-row block rather than at whole blocks (qx_gemv_chain's unit), so that the
 * CTAs finish together: the slices of a block split between CTAs are summed
 * in fp32 per CTA and then in CTA order, so the results are deterministic and
 * within fp32 rounding of qx_gemv_chain's, and equal bit for bit between the
 * one-launch and the QX_GEMV_SEPARATE forms.
 * workspace: caller-owned device memory, 256-byte aligned, of at least
 * qx_gemv_fused_workspace() bytes, all zero before the first call: every
 * completed call leaves its counters zero (zero it again after
 * QX_ERR_TIMEOUT).  Calls that may run at the same time need separate
 * workspaces.  flags: 0, QX_GEMV_PDL, QX_GEMV_SEPARATE or both.  Errors: those
 * of qx_gemv_chain; INVALID_ARG (workspace NULL or too small), ALIGNMENT
 * (workspace). */
qx_status qx_gemv_fused(const qx_gemv_group *groups, int32_t ngroups, int32_t batch, int32_t y_dtype,
                        int32_t flags, void *workspace, size_t workspace_bytes, void *stream);

/* qx_decode_step with the groups run by qx_gemv_fused (same workspace rules). */
qx_status qx_decode_step_fused(const qx_copy *in, int32_t nin, const qx_gemv_group *groups, int32_t ngroups,
                               int32_t batch, int32_t y_dtype, int32_t flags, void *workspace,
                               size_t workspace_bytes, const qx_copy *out, int32_t nout, int32_t sync,
                               void *stream);

/* Prefill matmul Y = X W_hat^T (Table 2 "Prefill") on the tcgen05 tensor cores:
 * W_hat tiles are dequantized into shared memory and multiplied in fp16 with
 * fp32 accumulation in tensor memory, 256 tokens per tile (16 when m <= 16).
 * X: device fp16 [m][k] row-major, 16-byte aligned; Y: device fp16 [m][n]
 * row-major, 4-byte aligned; m >= 1.  One CTA per tile: no workspace. */
qx_status qx_gemm(const qx_packed *p, const void *X, int64_t m, void *Y, void *stream);

/* Flags of qx_gemm_splitk. */
enum {
    /* Launch with programmatic dependent launch: the kernel may start, and
     * stream and dequantize this call's weights, while the previous kernel in
     * the stream is still running; it waits for that kernel before reading X
     * or writing Y and the workspace.  Set it only when the previous kernel
     * does not write this call's weights. */
    QX_GEMM_PDL = 1
};

/* Bytes of workspace qx_gemm_splitk needs for an n x k matrix of `recipe` and
 * m rows of X on the current device (host-only call; 0 when the call will not
 * split k).  Same shape rules as qx_packed_size; m >= 1. */
qx_status qx_gemm_splitk_workspace(int64_t n, int64_t k, int64_t m, const qx_recipe *recipe,
                                   size_t *bytes);

/* Host only: the plan qx_gemm_splitk takes for an n x k matrix and m rows of X
 * on a GPU with num_sms SMs -- tokens per tile (16, 64 or 256), k splits per
 * tile (1..16) and workspace bytes (0 when splits = 1).  The plan depends only
 * on these numbers.  Errors: INVALID_ARG (NULL, a size < 1), UNSUPPORTED (k
 * not a multiple of 128, or n, k, m beyond the library's limits). */
qx_status qx_gemm_splitk_plan(int64_t n, int64_t k, int64_t m, int32_t num_sms, int32_t *token_tile,
                              int32_t *splits, size_t *bytes);

/* qx_gemm with the contraction split along k (at 128-weight boundaries) when
 * the tiles alone would leave SMs idle -- the decode case (m <= 16: 16-token
 * tiles, so this is also the tensor-core decode matmul for batches of 1..16)
 * and short prefills (64-token tiles split along k, or 256-token tiles,
 * whichever the tile count favours).  Each split stores an fp32 partial tile to `workspace`;
 * the last split of a tile to finish sums the partials in split order (the
 * result does not depend on timing) and writes Y.  Same X, Y, m rules as
 * qx_gemm.
 * workspace: caller-owned device memory, 256-byte aligned, of at least
 * qx_gemm_splitk_workspace() bytes (may be null when that is 0).  Its first
 * 64 KiB hold counters, which must be zero before the first call: fill the
 * whole buffer with zeros once; every completed call, whatever its shape,
 * leaves them zero again.  After a call that ends
 * in QX_ERR_TIMEOUT, zero it again.  Calls that may run at the same time need
 * separate workspaces.  Returns QX_ERR_INVALID_ARG if the workspace is
 * missing or too small, QX_ERR_ALIGNMENT if it is misaligned.
 * flags: 0 or QX_GEMM_PDL. */
qx_status qx_gemm_splitk(const qx_packed *p, const void *X, int64_t m, void *Y, void *workspace,
                         size_t workspace_bytes, int32_t flags, void *stream);

/* qx_gemm_splitk for callers that cannot allocate device memory: it allocates
 * nothing and takes no workspace.  The partial tiles go to a scratch array of
 * 4 MiB that the library holds in static device memory, one per device (64 KiB
 * of counters, then room for 504 split units of 16 tokens); its address is
 * looked up once per device.  Each call clears the counters it uses on
 * `stream` before the launch.  Same arguments, results and rules as
 * qx_gemm_splitk otherwise; calls on one device must not run at the same time
 * (they share the scratch).  Returns QX_ERR_UNSUPPORTED when the split plan
 * needs more than the scratch holds (qx_gemm_splitk_workspace() > 4 MiB). */
qx_status qx_gemm_splitk_noalloc(const qx_packed *p, const void *X, int64_t m, void *Y, void *stream);

/* 8-bit per-token activations (Table 2: "8-bit RTN per-token quantization for
 * the activation tensors"; Table 1: W3A8), for qx_gemv_a8.  For each token b
 * (row of x): s_b = fp32(max_k |x[b][k]| / 127) and q[b][k] = clamp(rint(x / s_b),
 * -127, 127) in IEEE fp32 (q = 0 when s_b = 0); bit-exact with the CPU oracle.
 * x: device fp16 [batch][k], finite; q: device int8 [batch][k], 16-byte
 * aligned; scales: device fp32 [batch].  batch 1..2^24 (decode batches and
 * prefill token counts alike), k a multiple of 16 up to 2^20. */
qx_status qx_quantize_act(const void *x, int32_t batch, int64_t k, void *q, void *scales, void *stream);

/* W.A8 prefill activations: the tensor cores take fp16 operands, so the int8
 * codes of qx_quantize_act enter the matmul as x_hat[b][k] = fp16(fp32(s_b *
 * q[b][k])), one IEEE fp32 product then a round to nearest even; bit-exact
 * with the CPU oracle.  Y = x_hat W_hat^T is then qx_gemm (or qx_gemm_splitk,
 * qx_q4x_gemm) on x_hat: the W.A8 prefill, for any weight format.
 * q: device int8 [m][k], 16-byte aligned; scales: device fp32 [m]; x_hat:
 * device fp16 [m][k], 16-byte aligned.  m 1..2^24, k a multiple of 16 up to
 * 2^20.  Asynchronous on `stream`.  Errors (nothing launched): INVALID_ARG
 * (NULL, m < 1, k < 1), UNSUPPORTED (k not a multiple of 16, k > 2^20,
 * m > 2^24), ALIGNMENT (q or x_hat not 16-byte, scales not 4-byte aligned). */
qx_status qx_dequant_act(const void *q, const void *scales, int64_t m, int64_t k, void *x_hat, void *stream);

/* W.A8 decode matmul for uniform weights: y[b][n] = s_b * sum_g s_g *
 * sum_{k in g} (q_w - z) q[b][k], the group sums exact integers (dp4a), the
 * scales applied in fp32.  q, scales: the output of qx_quantize_act for this
 * matrix's k; y: device [batch][n] of y_dtype, 4-byte aligned.  Non-uniform
 * (LUT) recipes have no integer form: QX_ERR_UNSUPPORTED. */
qx_status qx_gemv_a8(const qx_packed *p, const void *q, const void *scales, int32_t batch, void *y,
                     int32_t y_dtype, void *stream);

/* Per-matrix recipe selection (Sections 2.2-2.3: uniform or non-uniform per
 * matrix by the Frobenius norm of the quantization error; bit-widths chosen
 * per layer).  For each of the `count` candidate recipes (1..16) whose bits per
 * weight (8 x packed bytes / (n k), returned in bpw[i]) are at most max_bpw
 * (every candidate when max_bpw <= 0), W is quantized and dequantized on the
 * device and E_i = sum (w - w_hat)^2 is taken exactly: sq_error[2i] (low word)
 * and sq_error[2i+1] hold E_i * 2^48, an integer; both words are all ones for a
 * candidate over the budget.  *chosen = the eligible candidate with the
 * smallest E_i, ties to the smaller bpw, then to the earlier index; -1 when
 * none is eligible.
 * A candidate of kind QX_Q4X (bits 4, group_size 64, lloyd_iters 0..1000 as
 * the learner's step limit, else UNSUPPORTED / INVALID_ARG) is quantized by
 * qx_q4x_quantize and dequantized by qx_q4x_dequant; its bytes are the four
 * Q4X buffers of qx_q4x_size, codebooks included.
 * W: device fp16 [n][k], 16-byte aligned, as for qx_quantize.  candidates,
 * chosen, sq_error (2 count words), bpw (count): host memory.  workspace:
 * device memory, 256-byte aligned, of at least qx_select_workspace() bytes.
 * The call synchronizes `stream`.  Returns QX_ERR_NONFINITE if W holds NaN or
 * Inf (the device status word keeps the flag). */
qx_status qx_select_workspace(int64_t n, int64_t k, const qx_recipe *candidates, int32_t count, size_t *bytes);
qx_status qx_select_recipe(const void *W, int64_t n, int64_t k, const qx_recipe *candidates, int32_t count,
                           double max_bpw, void *workspace, size_t workspace_bytes, int32_t *chosen,
                           uint64_t *sq_error, double *bpw, void *stream);

/* Q4X shared-codebook matrices (Section 3.2, Fig. 3a/3b; Table 2 "Q4X
 * W4A8G64", 4.28 bits per weight).  Groups of 64 consecutive weights along k;
 * each group has an fp16 scale s = max|w| and a 2-bit index b naming one of
 * four codebooks of 16 fp16 levels in [-1, 1], learned per matrix; every
 * weight has a 4-bit code q.
 *   codes     : uint8 [n][k/2], the 4-bit code layout of the header comment
 *   scales    : fp16 [n][k/64]
 *   books     : uint8 [n][ceil(k/256)]; group j's index in bits 2(j%4) and
 *               2(j%4)+1 of byte j/4; a row's unused high bits are zero
 *   codebooks : fp16 [4][16], each ascending
 * Dequantized weight: w_hat = fp16_rn((float)s * (float)codebooks[b][q]).
 * Shapes: n >= 1, k a multiple of 64, n*k at most 2^31.  All four pointers
 * are device memory; codes 16-byte aligned, scales and codebooks 2-byte. */
typedef struct qx_q4x {
    int64_t n, k;
    void *codes;
    void *scales;
    void *books;
    void *codebooks;
} qx_q4x;

typedef struct qx_q4x_sizes {
    uint64_t codes, scales, books, codebooks;
} qx_q4x_sizes;

/* Host only: byte sizes of the four Q4X buffers of an n x k matrix, and of the
 * workspace qx_q4x_quantize needs (about 42 bytes per group plus 42 MB:
 * per-group histograms, the value histograms of the four books).
 * Errors: INVALID_ARG (NULL, n < 1, k < 1), UNSUPPORTED (k not a multiple of
 * 64, n*k above 2^31). */
qx_status qx_q4x_size(int64_t n, int64_t k, qx_q4x_sizes *out);
qx_status qx_q4x_workspace(int64_t n, int64_t k, size_t *bytes);

/* Learn the four codebooks of W (device fp16 [n][k] = out->n x out->k,
 * 16-byte aligned) and code it into *out, bit-identical to the CPU oracle:
 * s = max|w| per group; U = rint(w / s 2^20) (float64); a 32-bin histogram of
 * U per group; k-means with 4 centres over the histograms (start: the groups
 * at ranks floor((2j+1) L / 8) by sum U^2, then position; float64 distances
 * in bin order, ties to the lower centre; exact integer means); each book's
 * 16 levels by Lloyd-Max over its groups' U (quantile start, ties to the lower
 * level, exact integer cell sums); codebook = fp16(level / 2^20); codes = the
 * nearest of the 16 fp16 candidates (ties to the lower).  Both iterations stop
 * when an assignment repeats, after at most `iters` (0..1000) steps.
 * workspace: device memory, 256-byte aligned, of at least qx_q4x_workspace()
 * bytes; the call zero-fills what it needs.  Asynchronous on `stream`; NaN or
 * Inf in a group sets QX_ERR_NONFINITE in the device status and codes that
 * group as all zero. */
qx_status qx_q4x_quantize(const void *W, int32_t iters, const qx_q4x *out, void *workspace,
                          size_t workspace_bytes, void *stream);

/* Dequantize into W_out (device fp16 [n][k], 16-byte aligned), bit-exact with
 * the formula above. */
qx_status qx_q4x_dequant(const qx_q4x *p, void *W_out, void *stream);

/* Decode matmul y = x W_hat^T for a Q4X matrix: x device fp16 [batch][k],
 * 16-byte aligned; y device [batch][n] of y_dtype, 4-byte aligned; batch
 * 1..16.  w_hat exactly as above.  When k is a multiple of 128 (and at most
 * 32768) the codes are decoded in registers from TMA-staged tiles, as qx_gemv
 * does (Section 2.4): for one or two rows of x the products of the codebook
 * levels (in [-1, 1]) with x and their sums over 8 weight pairs are formed in
 * fp16, then summed in fp32 and multiplied by the group's scale (s * sum
 * CB[q] x, not sum w_hat x: they differ by the rounding of w_hat); for 3..16
 * rows the products of w_hat itself are summed in fp32 on the tensor cores.
 * Otherwise the products of w_hat and their sums over 16 consecutive pairs are
 * formed in fp16, then summed in fp32.  fp16 intermediates must stay within
 * its range (|.| < 65504).  A matrix's results do not depend on the other
 * matrices of a qx_q4x_gemv_multi call. */
qx_status qx_q4x_gemv(const qx_q4x *p, const void *x, int32_t batch, void *y, int32_t y_dtype, void *stream);

/* Several Q4X decode matmuls in one launch: y[i] = x[i] W_hat_i^T, i < count
 * (count 1..8), each matrix with its own shape and codebooks; x[i], y[i] have
 * the layout and alignment of qx_q4x_gemv and are passed in host arrays of
 * `count` device pointers.  One persistent grid strides over the rows of all
 * matrices (e.g. the q, k, v or gate, up projections of a decoder layer,
 * which share x), so the launch cost is paid once for the group. */
qx_status qx_q4x_gemv_multi(const qx_q4x *mats, int32_t count, const void *const *x, int32_t batch,
                            void *const *y, int32_t y_dtype, void *stream);

/* Prefill matmul Y = X W_hat^T for a Q4X matrix on the tcgen05 tensor cores,
 * as qx_gemm: W_hat tiles are dequantized into shared memory (the four
 * codebooks staged there once per CTA, w_hat exactly as above) and multiplied
 * in fp16 with fp32 accumulation.  X: device fp16 [m][k], 16-byte aligned;
 * Y: device fp16 [m][n], 2-byte aligned; m >= 1; k a multiple of 128. */
qx_status qx_q4x_gemm(const qx_q4x *p, const void *X, int64_t m, void *Y, void *stream);

/* qx_q4x_gemm with the contraction split along k when the tiles alone leave
 * SMs idle, exactly as qx_gemm_splitk (same plan, workspace rules, PDL flag and
 * split-order sum).  qx_q4x_gemm_splitk_workspace gives the workspace bytes
 * on the current device (0: no split). */
qx_status qx_q4x_gemm_splitk_workspace(int64_t n, int64_t k, int64_t m, size_t *bytes);
qx_status qx_q4x_gemm_splitk(const qx_q4x *p, const void *X, int64_t m, void *Y, void *workspace,
                             size_t workspace_bytes, int32_t flags, void *stream);

/* Failure-detection self-test.  Launches one CTA on `stream` whose bounded
 * wait (the mbarrier wait of the decode and prefill pipelines) is for a phase
 * that nothing completes.  After limit_us microseconds (1..1000000) it gives
 * up, records QX_ERR_TIMEOUT in the device status word and returns, leaving
 * the context usable; qx_get_device_status() then returns QX_ERR_TIMEOUT. */
qx_status qx_selftest_wait_timeout(int32_t limit_us, void *stream);

/* Library infrastructure, no passage of the paper (which describes no error
 * handling): synchronize `stream`, then return and clear the current device's
 * status word (QX_OK, QX_ERR_NONFINITE or QX_ERR_TIMEOUT).  Returns
 * QX_ERR_CUDA if the synchronization itself fails. */
qx_status qx_get_device_status(void *stream);

/* Library infrastructure, no passage of the paper: a static, NUL-terminated
 * description of a status code. */
const char *qx_status_string(qx_status s);

/* Name of the last CUDA error an entry point of this thread turned into
 * QX_ERR_CUDA (a static string; "no error" if none). */
const char *qx_last_error_string(void);

/* Library version as major*10000 + minor*100 + patch. */
int32_t qx_version(void);

#ifdef __cplusplus
}
#endif

#endif /* QX_H */
