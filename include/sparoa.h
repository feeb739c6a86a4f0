/*
 * libsparoa -- sparsity/intensity-dispatched DNN operators on one GB300 (sm_103a).
 *
 * For each convolution or fully connected operator the library measures the
 * input's zero fraction (Eq. 1 of the SparOA paper, arXiv 2511.19457, Sec. 3.1)
 * and its computational intensity (Eq. 2, Sec. 3.1, taken as FLOPs per byte of
 * input activation), compares both with two thresholds (Sec. 2.2 quadrants,
 * Sec. 3 threshold rule; here plain parameters), and runs the operator either
 * on a zero-skipping kernel (Sec. 2.1: zero-valued products are skipped without
 * changing the output) or on a dense tensor-core kernel.  Depthwise
 * convolution, pooling and batch-norm/activation -- the memory-bound operators
 * of the paper's low-intensity quadrant (Sec. 2.2) -- have their own kernels.
 * Every kernel that writes a bf16 activation can also write the Eq. 1 count and
 * occupancy bitmaps of that activation, so the next operator's dispatch needs
 * no separate pass.
 *
 * Conventions for every entry point
 *   - Plain C ABI.  No exception crosses it; every call returns a status.  On
 *     failure the context keeps a message (sparoa_last_error).
 *   - Tensors are caller-owned DEVICE pointers (CUDA global memory of the
 *     context's device) unless a parameter says "host".  The library never frees
 *     caller memory.  Pointers passed to kernels that use TMA (x and W of
 *     sparoa_gemm, W of sparoa_conv2d) must be 16-byte aligned.
 *   - Activations are bf16, NHWC for convolutions and row-major [M, K] for FC.
 *     Conv weights are [C_out][k_h][k_w][C_in/groups] bf16; FC weights are
 *     [N][K] bf16 (and optionally the same values as [K][N]).  Bias, batch-norm
 *     parameters and FP32 outputs are fp32.
 *   - All work is enqueued on the context's CUDA stream and is asynchronous,
 *     except that a non-NULL host output (sparoa_stats*, sparoa_record*) makes
 *     the call wait for the stream before it returns.
 *   - Device-side failures (a bounded wait inside a kernel that ran out) are
 *     recorded in the context and reported as SPAROA_ERR_TIMEOUT by the next
 *     call that synchronises (any call with a host output, or sparoa_sync).
 */
#ifndef SPAROA_H
#define SPAROA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SPAROA_OK = 0,
    SPAROA_ERR_INVALID_ARG = 1,  /* null pointer, bad size, misaligned pointer  */
    SPAROA_ERR_UNSUPPORTED = 2,  /* valid request the library does not implement */
    SPAROA_ERR_OOM = 3,          /* workspace allocation failed                 */
    SPAROA_ERR_CUDA = 4,         /* a CUDA runtime/driver call failed           */
    SPAROA_ERR_TIMEOUT = 5       /* a kernel's bounded wait ran out             */
} sparoa_status;

typedef enum { SPAROA_BF16 = 0, SPAROA_F32 = 1 } sparoa_dtype;

/* Which kernel ran an operator. */
typedef enum {
    SPAROA_PATH_NONE = 0,       /* pooling / batch norm: no dispatch          */
    SPAROA_PATH_DENSE_TC = 1,   /* dense tcgen05 tensor-core kernel           */
    SPAROA_PATH_ZERO_SKIP = 2,  /* zero-skipping kernel                       */
    SPAROA_PATH_DEPTHWISE = 3   /* depthwise kernel (groups == channels)      */
} sparoa_path;

/* GELU (transformer MLPs) is computed in the tanh form of Hendrycks and
 * Gimpel, within about 1e-3 of the exact v * Phi(v). */
typedef enum {
    SPAROA_ACT_NONE = 0, SPAROA_ACT_RELU = 1, SPAROA_ACT_RELU6 = 2, SPAROA_ACT_GELU = 3
} sparoa_act;

typedef enum {
    SPAROA_OP_CONV2D = 1,       /* groups 1 (dispatched) or depthwise          */
    SPAROA_OP_FC = 2,           /* fully connected, input flattened to [M, K]  */
    SPAROA_OP_MAXPOOL = 3,      /* k x k max pool (kh, stride, pad)            */
    SPAROA_OP_AVGPOOL = 4,      /* global average pool, [N,H,W,C] -> [N,C]     */
    SPAROA_OP_BN_ACT = 5,       /* element-wise epilogue only                  */
    /* Vision-transformer operators (Sec. 6, Table 2: ViT-B16).  Tokens are the
     * W positions of an [N, 1, T, C] value; a token-wise linear layer is a 1x1
     * CONV2D on it. */
    SPAROA_OP_LAYERNORM = 6,    /* per row over C; bn = fp32 [2][C] gamma, beta
                                   (nullable), bn_eps = epsilon; C % 8 == 0   */
    SPAROA_OP_ATTENTION = 7,    /* input rows q | k | v (3 D = 3 heads hd
                                   values), groups = heads; output [.., D];
                                   T <= 512, hd 16, 32 or 64                 */
    SPAROA_OP_TOKENS = 8,       /* [N, h, w, D] -> [N, 1, 1 + h w, D]: row 0
                                   weight (bf16 [D], the class token), rows
                                   1.. the positions; + bias (fp32 position
                                   table [1 + h w][D]); D % 8 == 0           */
    SPAROA_OP_SELECT = 9        /* [N, H, W, D] -> [N, 1, 1, D]: position
                                   `pad` of H x W (the class token: 0)       */
} sparoa_op_kind;

/*
 * Thresholds of the dispatch rule (Sec. 3: a sparsity threshold s and an
 * intensity threshold c per operator; the paper predicts them, this library
 * takes them as parameters).  Rule, evaluated in IEEE double:
 *     zero-skip  if (double)(numel - nnz) >= s_thr * (double)numel
 *     dense      else if intensity >= c_thr
 *     zero-skip  otherwise
 * intensity_mode 0: intensity = FLOPs per input byte (default);
 *                1: intensity = the Eq. 2 count K_h*K_w*C_in*C_out*H_out*W_out.
 * force_path 0 = rule, 1 = always dense, 2 = always zero-skip.
 * Passing NULL means { s_thr = 0.5, c_thr = 32, mode 0, force 0 }.
 */
typedef struct {
    double s_thr;
    double c_thr;
    int32_t intensity_mode;
    int32_t force_path;
} sparoa_thresholds;

/* Host-side record of one operator: Eq. 1 numbers of its input, Eq. 2 work,
 * the input shape features of Sec. 3.1 and the path taken. */
typedef struct {
    uint64_t numel;          /* n(O) of Eq. 1                               */
    uint64_t nnz;            /* c(O) of Eq. 1                               */
    double sparsity;         /* rho = 1 - c(O)/n(O)                          */
    uint64_t flops;          /* 2*N*H_out*W_out*C_out*(C_in/groups)*K_h*K_w  */
    uint64_t macs_eq2;       /* Eq. 2 literally                              */
    uint64_t input_bytes;    /* numel * sizeof(bf16)                         */
    double flops_per_byte;   /* flops / input_bytes                          */
    int32_t B, C_in, H, W;   /* input features of Sec. 3.1                   */
    int32_t path;            /* sparoa_path                                  */
    int32_t reserved;
} sparoa_stats;

/*
 * Device-resident Eq. 1 count and occupancy bitmaps of a bf16 tensor viewed as
 * a matrix [R, C] (R = N*H*W rows of an NHWC tensor, C = channels; or [M, K]).
 * Let T = ceil(C/64), W64 = ceil(T/64), RB = ceil(R/128), C32 = ceil(C/32):
 *   nnz[1]               number of elements whose bf16 pattern is not +0/-0
 *   col_nnz[C]           non-zeros per column
 *   tile_nnz[T]          non-zeros per 64-column tile
 *   row_bm[R*W64]        bit t%64 of word t/64 of row r: row r has a non-zero in
 *                        columns [64t, 64t+64)
 *   blk_mask[RB*C32]     bit c%32 of word c/32 of block b: column c has a
 *                        non-zero in rows [128b, 128b+128)
 * Bits past column C-1 or row R-1 are zero.  The whole block is one caller
 * buffer of sparoa_occupancy_bytes(R, C) bytes carved by sparoa_occupancy_init;
 * a producing call clears it on its stream before it writes.
 */
typedef struct {
    uint64_t *nnz;
    uint32_t *col_nnz;
    uint32_t *tile_nnz;
    uint64_t *row_bm;
    uint32_t *blk_mask;
    int64_t R, C;
    uint64_t bytes;          /* size of the block starting at nnz            */
} sparoa_occupancy;

/* Epilogue applied per output channel c to the fp32 accumulator v:
 *   v += bias[c];  v = (v - mean[c]) * gamma[c] / sqrt(var[c] + eps) + beta[c];
 *   v += residual (bf16, same shape as the output);  v = act(v).
 * Any pointer may be NULL (term skipped).  bn is fp32 [4][C_out]:
 * rows gamma, beta, mean, var. */
typedef struct {
    const float *bias;
    const float *bn;
    float bn_eps;
    int32_t act;
    const void *residual;
} sparoa_epilogue;

/* One operator of a graph (sparoa_run_graph).  Values are numbered: 0 is the
 * graph input, i+1 is the output of op i.  Ops must be in topological order
 * (Sec. 4.1: operators run in layer execution order): input and residual refer
 * to values < i+1. */
typedef struct {
    int32_t kind;            /* sparoa_op_kind                               */
    int32_t input;           /* value index of the input                      */
    int32_t residual;        /* value index added before the activation, or -1 */
    int32_t c_in, c_out;     /* channels (FC: K and N)                        */
    int32_t kh, kw, stride, pad, groups;
    int32_t act;             /* sparoa_act                                    */
    int32_t reserved;
    const void *weight;      /* device bf16, see conventions                  */
    const void *weight_kn;   /* FC only, optional [K][N] copy of the weights  */
    const float *bias;       /* device fp32 [c_out] or NULL                   */
    const float *bn;         /* device fp32 [4][c_out] or NULL                */
    float bn_eps;
    float reserved2;
    sparoa_thresholds thr;
} sparoa_op;

/* Per-operator result of sparoa_run_graph. */
typedef struct {
    sparoa_stats stats;      /* of the op's input; path taken                 */
    const void *output;      /* device pointer of the op's bf16 output inside
                                the context workspace; valid until the next
                                sparoa_run_graph on this context or destroy   */
    int64_t out_shape[4];    /* N, H, W, C  (FC / avg pool: M, 1, 1, C)       */
    const sparoa_occupancy *out_occ; /* occupancy of that output (same life)   */
} sparoa_record;

typedef struct sparoa_ctx sparoa_ctx;

/* ------------------------------------------------------------------------ */
/* Context                                                                   */
/* ------------------------------------------------------------------------ */

/* Create a context on CUDA device `device` that enqueues on `stream` (a
 * cudaStream_t; NULL = the legacy default stream).  The context owns only its
 * workspace (device scratch for statistics, padding and graph activations),
 * grown on demand and freed by sparoa_destroy.
 * Errors: INVALID_ARG (out == NULL, bad device), CUDA, OOM. */
sparoa_status sparoa_create(sparoa_ctx **out, int device, void *stream);

/* Wait for the context's stream, then free its workspace.  NULL is a no-op. */
sparoa_status sparoa_destroy(sparoa_ctx *ctx);

/* Change the stream later calls enqueue on. */
sparoa_status sparoa_set_stream(sparoa_ctx *ctx, void *stream);

/* Launch overlap (default on): each kernel of a call is launched with CUDA's
 * programmatic stream serialization, so that its on-chip prologue (barrier
 * initialisation, tensor-memory allocation) runs while the kernel before it
 * on the stream finishes.  Before the previous grid has completed a kernel
 * writes no global memory and reads only inputs that an earlier kernel of the
 * same call has already waited for (so they are complete), so results do not
 * depend on this setting.  enable = 0 launches plainly.
 * Errors: INVALID_ARG (ctx == NULL). */
sparoa_status sparoa_set_overlap(sparoa_ctx *ctx, int32_t enable);

/* Wait for the stream; report (and clear) a device-side timeout. */
sparoa_status sparoa_sync(sparoa_ctx *ctx);

/* Wait for the stream and write to *path the path that the last sparoa_gemm
 * or sparoa_conv2d call on this context took (SPAROA_PATH_DENSE_TC /
 * SPAROA_PATH_ZERO_SKIP / SPAROA_PATH_DEPTHWISE, as its kernel recorded it on
 * the device: Sec. 3's rule), without the call's full statistics record.
 * Errors: INVALID_ARG (ctx or path NULL), CUDA, TIMEOUT as sparoa_sync. */
sparoa_status sparoa_last_path(sparoa_ctx *ctx, int32_t *path);

/* Testing hooks for the failure paths (the paper has no counterpart).
 *
 * sparoa_set_wait_limit: SM clock cycles after which a tensor-core kernel's
 * bounded waits give up (0 = the default, about a second).  A wait that runs
 * out records an error bit in the context and lets every CTA unwind: it waits
 * (bounded again) for the copies and MMAs it already issued, frees its tensor
 * memory and exits; the next synchronising call returns SPAROA_ERR_TIMEOUT and
 * the context stays usable.
 * sparoa_set_fault: 1 = the tensor-core kernels' MMA issuer withholds its
 * signal for the first accumulator of each CTA until the code is set back to
 * 0, so that the epilogue's bounded wait runs out (no fault, trap or endless
 * loop on the GPU); 2 = the next workspace allocation of the context fails
 * (SPAROA_ERR_OOM), once; 0 = off.
 * Errors: INVALID_ARG (ctx NULL, negative cycles, unknown code). */
sparoa_status sparoa_set_wait_limit(sparoa_ctx *ctx, int64_t cycles);
sparoa_status sparoa_set_fault(sparoa_ctx *ctx, int32_t code);

/* Static description of a status code. */
const char *sparoa_status_str(sparoa_status s);

/* Message of the last failure on this context ("" if none).  Owned by ctx. */
const char *sparoa_last_error(const sparoa_ctx *ctx);

/* ------------------------------------------------------------------------ */
/* Occupancy buffers                                                          */
/* ------------------------------------------------------------------------ */

/* Bytes of the occupancy block of a [R, C] tensor (layout above). */
uint64_t sparoa_occupancy_bytes(int64_t R, int64_t C);

/* Carve `dev_buf` (device, >= sparoa_occupancy_bytes(R, C) bytes, 16-byte
 * aligned) into `out`.  Host-only; touches no device memory.
 * Errors: INVALID_ARG. */
sparoa_status sparoa_occupancy_init(void *dev_buf, uint64_t bytes, int64_t R, int64_t C,
                                    sparoa_occupancy *out);

/* ------------------------------------------------------------------------ */
/* Operators                                                                  */
/* ------------------------------------------------------------------------ */

/*
 * Eq. 1 statistics of a bf16 tensor x viewed as [R = N*H*W, C] (Sec. 3.1:
 * sparsity from the count of non-zero elements), plus the occupancy bitmaps.
 *   occ       device outputs (nullable: then only host_out is produced, using
 *             context scratch)
 *   consumer  the operator that will read x (nullable).  Gives Eq. 2 work,
 *             FLOPs per input byte and the path the rule picks; NULL leaves
 *             flops = 0 and path = NONE.
 *   host_out  host record (nullable; synchronises)
 * Errors: INVALID_ARG (x NULL with numel > 0, negative sizes), CUDA, OOM.
 */
sparoa_status sparoa_op_stats(sparoa_ctx *ctx, const void *x, int64_t N, int64_t H, int64_t W,
                              int64_t C, const sparoa_op *consumer, const sparoa_occupancy *occ,
                              sparoa_stats *host_out);

/*
 * Fully connected operator with threshold dispatch:
 *   y[M, N] = epilogue( x[M, K] * W[N, K]^T )
 * x_occ: occupancy of x if already known (e.g. written by the producer's
 * epilogue); NULL = measured here into context scratch.  The path is decided
 * on the device from x's non-zero count, so no host synchronisation happens
 * unless host_out is given.  Dense path: tcgen05 tensor-core GEMM.  Zero-skip
 * path: for M <= 128 with W_kn given, a column-compacting kernel that reads
 * only the rows of W_kn whose activation column is occupied; otherwise a
 * tcgen05 GEMM that stages only the 32-wide K blocks occupied in each 128-row
 * block of x.
 *   W_kn    optional [K][N] copy of W (nullable)
 *   y_dtype SPAROA_BF16 or SPAROA_F32
 *   y_occ   occupancy of y to write (nullable; bf16 y only)
 * Requirements: K % 8 == 0, N % 8 == 0 (TMA row pitch), x and W 16-byte aligned.
 * Errors: INVALID_ARG, UNSUPPORTED (y_occ with F32 output), CUDA, OOM.
 */
sparoa_status sparoa_gemm(sparoa_ctx *ctx, const void *x, int64_t M, int64_t K, const void *W,
                          const void *W_kn, int64_t N, const sparoa_epilogue *ep,
                          const sparoa_thresholds *thr, void *y, int32_t y_dtype,
                          const sparoa_occupancy *x_occ, const sparoa_occupancy *y_occ,
                          sparoa_stats *host_out);

/*
 * Split execution of one FC operator (the single-GPU analogue of the paper's
 * co-execution, Sec. 5.1 and its aggregation equation): rows [0, Ms) of x run
 * through the zero-skip kernel and rows [Ms, M) through the dense tensor-core
 * kernel, Ms = xi * M rounded to whole 128-row blocks.  The two parts are
 * launched on two streams of the context (forked from and joined back into
 * its stream, so stream capture records both) and write disjoint rows of y;
 * y_occ, when given, is assembled from both parts.  The result equals that of
 * sparoa_gemm up to the floating-point summation order of the chosen kernels.
 *   xi      fraction of the rows for the zero-skip kernel, in [0, 1]
 * Other arguments and requirements as sparoa_gemm (no host record).
 * Errors: INVALID_ARG (also xi outside [0, 1]), UNSUPPORTED, CUDA, OOM.
 */
sparoa_status sparoa_gemm_split(sparoa_ctx *ctx, const void *x, int64_t M, int64_t K, const void *W,
                                const void *W_kn, int64_t N, const sparoa_epilogue *ep, double xi,
                                void *y, int32_t y_dtype, const sparoa_occupancy *x_occ,
                                const sparoa_occupancy *y_occ);

/*
 * 2-D convolution with threshold dispatch, NHWC:
 *   y[N, Ho, Wo, C_out] = epilogue( conv(x[N, H, W, C_in], w) ),
 *   Ho = (H + 2*pad - kh)/stride + 1,  Wo likewise.
 * groups == 1: dispatched between a dense tcgen05 implicit-GEMM kernel and the
 * same kernel with zero-skipping of (tap, channel-block) K slices whose 128
 * shifted input rows are all unoccupied.  groups == C_in == C_out: the
 * depthwise kernel (path DEPTHWISE).  Other groups: UNSUPPORTED.
 * C_in that is not a multiple of 8 is zero-padded to one in context scratch.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA, OOM.
 */
sparoa_status sparoa_conv2d(sparoa_ctx *ctx, const void *x, int64_t N, int64_t H, int64_t W,
                            int64_t C_in, const void *w, int64_t C_out, int32_t kh, int32_t kw,
                            int32_t stride, int32_t pad, int32_t groups,
                            const sparoa_epilogue *ep, const sparoa_thresholds *thr, void *y,
                            const sparoa_occupancy *x_occ, const sparoa_occupancy *y_occ,
                            sparoa_stats *host_out);

/* k x k max pooling, NHWC, padded positions ignored.  C % 8 == 0.
 * Errors: INVALID_ARG, CUDA. */
sparoa_status sparoa_maxpool2d(sparoa_ctx *ctx, const void *x, int64_t N, int64_t H, int64_t W,
                               int64_t C, int32_t k, int32_t stride, int32_t pad, void *y,
                               const sparoa_occupancy *y_occ);

/* Global average pooling [N, H, W, C] -> [N, C] (mean over H*W).  C % 8 == 0.
 * Errors: INVALID_ARG, CUDA. */
sparoa_status sparoa_avgpool_global(sparoa_ctx *ctx, const void *x, int64_t N, int64_t H,
                                    int64_t W, int64_t C, void *y,
                                    const sparoa_occupancy *y_occ);

/* Element-wise epilogue (bias, batch norm, residual, activation) over [R, C].
 * C % 8 == 0.  Errors: INVALID_ARG, CUDA. */
sparoa_status sparoa_bn_act(sparoa_ctx *ctx, const void *x, int64_t R, int64_t C,
                            const sparoa_epilogue *ep, void *y, const sparoa_occupancy *y_occ);

/* Layer normalisation of x [R, C] (bf16) over C (Sec. 3.2's LN): per row
 * (x - mean) / sqrt(biased variance + eps), then gamma * . + beta.
 *   gamma_beta  device fp32 [2][C] or NULL (1, 0)
 *   y_occ       occupancy of y to write (nullable)
 * C % 8 == 0.  Errors: INVALID_ARG, CUDA. */
sparoa_status sparoa_layernorm(sparoa_ctx *ctx, const void *x, int64_t R, int64_t C,
                               const float *gamma_beta, float eps, void *y,
                               const sparoa_occupancy *y_occ);

/* Multi-head self-attention (Sec. 3.2's MHSA) of N sequences of T tokens:
 * qkv [N, T, 3 D] bf16 holds per token q | k | v, each heads x head_dim values
 * (D = heads head_dim); per head, y = softmax(Q K^T / sqrt(head_dim)) V with the
 * heads concatenated, y [N, T, D] bf16; tensor cores, fp32 softmax and
 * accumulation, the probabilities rounded to bf16 for the P V products.
 * T <= 512, head_dim 16, 32 or 64.  Errors: INVALID_ARG, UNSUPPORTED (sizes), CUDA. */
sparoa_status sparoa_attention(sparoa_ctx *ctx, const void *qkv, int64_t N, int64_t T,
                               int32_t heads, int32_t head_dim, void *y,
                               const sparoa_occupancy *y_occ);

/*
 * Run a topologically ordered operator list (Sec. 4.1 layer execution order;
 * Sec. 5.1 operator-by-operator execution) on one GPU.  The input x is bf16
 * NHWC [N, H, W, C].  For every conv/FC operator the path is chosen on the
 * device from the occupancy its producer wrote, so the walk never waits on the
 * host.  Intermediate activations live in the context workspace.
 *   y        device destination for the last operator's bf16 output (nullable)
 *   y_bytes  capacity of y in bytes (checked)
 *   records  host array of n_ops records (nullable; synchronises)
 * Errors: INVALID_ARG (bad indices, shapes that do not chain), UNSUPPORTED,
 * CUDA, OOM, TIMEOUT.
 */
sparoa_status sparoa_run_graph(sparoa_ctx *ctx, const sparoa_op *ops, int32_t n_ops,
                               const void *x, int64_t N, int64_t H, int64_t W, int64_t C, void *y,
                               uint64_t y_bytes, sparoa_record *records);

/*
 * Device workspace sparoa_run_graph needs for this operator list and input
 * shape, in bytes: occupancy blocks of every value, recorded paths, every
 * intermediate activation (bf16) and channel-padded copies.  Checks the list
 * exactly as sparoa_run_graph does; no device work.  This is the memory model
 * M(B) of the dynamic batching loop (Sec. 5.2, Algorithm 2).
 *   bytes  host output
 * Errors: INVALID_ARG, UNSUPPORTED (as sparoa_run_graph).
 */
sparoa_status sparoa_graph_workspace(sparoa_ctx *ctx, const sparoa_op *ops, int32_t n_ops,
                                     int64_t N, int64_t H, int64_t W, int64_t C, uint64_t *bytes);

/* ------------------------------------------------------------------------ */
/* Variant for callers that cannot allocate device memory                     */
/* ------------------------------------------------------------------------ */

/* Size of the library's static device scratch array used by
 * sparoa_gemm_noalloc (4 MiB; every GPU that loads the library holds it until
 * the process exits). */
#define SPAROA_NOALLOC_SCRATCH_BYTES (4u << 20)

/*
 * sparoa_gemm without any device allocation.  The paper has no counterpart:
 * this exists for callers that cannot call cudaMalloc -- plugins inside a
 * framework whose allocator owns the device memory, and loops with a memory
 * budget fixed at start-up.  It computes exactly what sparoa_gemm
 * computes with x_occ = y_occ = NULL, but needs no context: work goes to
 * `stream` (a cudaStream_t; NULL = legacy default stream) on the current
 * device, and the input's occupancy (the only scratch) lives in a static
 * device array of SPAROA_NOALLOC_SCRATCH_BYTES bytes, 256 of which hold
 * control words.
 *   - The first call on a device looks the array's address up with
 *     cudaGetSymbolAddress while that device is current and keeps it for the
 *     process: a device reset (cudaDeviceReset) after that first call is not
 *     supported.
 *   - Calls share the array and each clears the part it uses before writing;
 *     calls whose work overlaps on the GPU (other streams or host threads)
 *     race on it and must be serialised by the caller.
 *   - x [M, K], W [N, K], optional W_kn [K, N], y [M, N] as in sparoa_gemm.
 *   - host_out (nullable) synchronises `stream` and fills the record.
 * Errors: INVALID_ARG (as sparoa_gemm); UNSUPPORTED when the occupancy of a
 * [M, K] input (sparoa_occupancy_bytes(M, K)) exceeds the array minus 256
 * bytes, or a dimension exceeds 2^30; CUDA; TIMEOUT (host_out only).
 */
sparoa_status sparoa_gemm_noalloc(void *stream, const void *x, int64_t M, int64_t K,
                                  const void *W, const void *W_kn, int64_t N,
                                  const sparoa_epilogue *ep, const sparoa_thresholds *thr,
                                  void *y, int32_t y_dtype, sparoa_stats *host_out);

#ifdef __cplusplus
}
#endif
#endif /* SPAROA_H */
