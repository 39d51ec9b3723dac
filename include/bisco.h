/*
 * bisco.h -- C ABI of the GB300 (sm_103a) library for BiSCo-LLM binary
 * spherical coded linear layers (arxiv 2607.08643).
 *
 * The paper states the problem, not an API: a weight matrix is cut into
 * d-dimensional chunks, each chunk is stored as a bit-packed sign pattern of
 * its unit-sphere direction (Sec. III-C, Eq. 3), further stages code the
 * residual left by the earlier ones (Sec. III-D, Eq. 5-7), a small set of
 * input channels chosen by Eq. 8 is kept in 8 bits instead (Sec. III-E,
 * Eq. 10), and inference decodes the stages independently and sums them
 * (Sec. III-G, Eq. 12) before the linear map y = W x.  This library runs
 * that linear map straight from the coded bytes, without ever writing the
 * dense weight to memory.  Beside that path it takes the method's variants:
 * output rows as the protected channels, with the coupled gate/up/down set
 * of a gated MLP (Eq. 9); FP8 and BF16 protected payloads; the learned
 * decoder of Eq. 1 given as per-stage tables; the materialised weight; and
 * the optional low-rank compensation.
 *
 * Conventions for every entry point:
 *   - All pointers are caller-owned DEVICE memory unless stated otherwise;
 *     the library allocates nothing and keeps no state between calls other
 *     than a per-device error word.
 *   - Pointers must be 16-byte aligned, else BISCO_ERR_INVALID_ARG; the
 *     per-channel float weights g and caller-given index lists need 4.
 *   - Calls are asynchronous on `stream` (NULL = the legacy default stream).
 *     Argument errors are returned synchronously and nothing is launched.
 *     Errors found on the device (fp16 overflow in encode, an expired
 *     bounded wait) are latched in the device error word and returned by
 *     bisco_get_device_error().  No function aborts or prints.
 *   - bf16 / fp16 values are passed as their uint16 bit patterns.
 */
#ifndef BISCO_H
#define BISCO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t / CUstream. */
typedef struct CUstream_st *bisco_stream_t;

typedef enum {
    BISCO_OK = 0,
    BISCO_ERR_INVALID_ARG = 1,  /* bad size, NULL or misaligned pointer        */
    BISCO_ERR_UNSUPPORTED = 2,  /* valid but not implemented (d != 8)          */
    BISCO_ERR_RANGE = 3,        /* encode: non-finite weight, fp16 norm/scale overflow */
    BISCO_ERR_CUDA = 4,         /* a CUDA runtime call failed                  */
    BISCO_ERR_TIMEOUT = 5       /* a bounded device-side wait expired          */
} bisco_status;

/*
 * One coded linear layer W (N = out features x K = in features, the
 * row-major layout of a PyTorch Linear weight).  Storage follows the paper's
 * real-size accounting (Sec. III-A, Eq. 2: S_code + S_8bit + S_meta; there
 * are no decoder or LoRA parameters):
 *
 *   codes    [S][N][K/8]  uint8   S_code.  Byte c of row i in stage s is
 *                                 chunk c = input columns 8c..8c+7; bit k
 *                                 is element k, 1 = negative (sign(0) = +).
 *   norms    [S][N][K/8]  uint16  S_meta.  binary16 L2 norm of that stage's
 *                                 chunk target; the chunk decodes to
 *                                 (bit ? -1 : +1) * norm / sqrt(8).
 *   q8       [N][p_pad]   int8    S_8bit.  Protected column t of row i at
 *                                 q8[i*p_pad + t], p_pad = roundup(p, 16),
 *                                 padding zero.
 *   q8_scale [p]          uint16  binary16 per-column scale (Eq. 10 Q8).
 *   prot_idx [p]          int32   protected input columns, strictly ascending.
 *
 * The decoded weight is  What[i][j] = sum_s (+-) norm_s[i][j/8] / sqrt(8)
 * for j not protected, and q8_scale[t] * q8[i][t] for j = prot_idx[t].
 *
 * With protect_axis = 1 the protected channels are OUTPUT ROWS (Sec. III-E
 * Eq. 9: the gate/up rows of a gated MLP, coupled with the down columns):
 *   q8       [p][kp]      int8    protected row t at q8[t*kp + k],
 *                                 kp = roundup(K, 16), padding zero.
 *   q8_scale [p]          uint16  binary16 per-row scale, max_k |W_ik| / 127.
 *   prot_idx [p]          int32   protected output rows, strictly ascending.
 * Those rows decode to What[i][k] = q8_scale[t] * q8[t][k] (i = prot_idx[t]);
 * the encoder zeroes them in the stage target, so their chunks store norm 0
 * and sign byte 0.  0 <= p <= N.
 */
typedef struct {
    int32_t n_out;        /* N >= 1                                       */
    int32_t k_in;         /* K >= 8, K % 8 == 0                            */
    int32_t chunk_dim;    /* d; only 8 is supported                        */
    int32_t stages;       /* S in {1, 2, 3}                                */
    int32_t n_protected;  /* p: 0 <= p <= K (axis 0), 0 <= p <= N (axis 1) */
    int32_t protect_axis; /* 0 = input columns; 1 = output rows            */
    uint8_t *codes;
    uint16_t *norms;
    int8_t *q8;           /* the protected payload, in protect_format      */
    uint16_t *q8_scale;
    int32_t *prot_idx;
    int32_t protect_format; /* BISCO_PROT_*: the protected payload's type */
} bisco_layer;

/*
 * Protected payload formats (the paper's protected-format ablation compares
 * INT8, FP8 E4M3, FP8 E5M2 and BF16 for the protected channels).  INT8 is
 * Eq. 10 as above.  For FP8 the per-column scale is
 * fp16(max_i |W_ij| / F), F the format's largest finite value (448 for
 * E4M3, 57344 for E5M2), and q = fp8(W_ij / scale) rounded to nearest, ties
 * to even, with gradual underflow; a quotient that rounds past F takes F
 * (saturation).  The q8 buffer then holds FP8 bytes in the same [N][p_pad]
 * layout (E4M3: bias 7, no infinities; E5M2: bias 15).  For BF16 the
 * payload is the weight itself, scale 1.0, and the buffer is [N][p_pad]
 * uint16 (twice the bytes).  On protected rows (protect_axis 1) the same
 * per-channel rules apply with the row as the channel: q [p][kp] elements
 * of the format, one scale per row.  The decode kernels run the binary
 * spherical stages without the protected set and then, in a second kernel,
 * replace each protected column's decoded value by scale * value(q) (or
 * overwrite each protected row).
 */
#define BISCO_PROT_INT8 0
#define BISCO_PROT_E4M3 1
#define BISCO_PROT_E5M2 2
#define BISCO_PROT_BF16 3

/* ABI version of this header (major * 100 + minor). */
#define BISCO_ABI_VERSION 107
int32_t bisco_abi_version(void);

/* Static string for a status code (never NULL). */
const char *bisco_status_string(int32_t status);

/*
 * Byte sizes of the five buffers of one layer, in the order codes, norms,
 * q8, q8_scale, prot_idx (Sec. III-A, Eq. 2).  Host-only, no device access.
 * Returns INVALID_ARG for N < 1, K < 8, K % 8 != 0, S not in 1..3, p out of
 * [0, K] or out_bytes == NULL; UNSUPPORTED for d != 8.
 */
bisco_status bisco_encoded_sizes(int32_t N, int32_t K, int32_t d, int32_t S,
                                 int32_t p, size_t out_bytes[5]);

/*
 * Byte sizes of the five buffers of the layer *L describes (its sizes,
 * protect_axis and protect_format; the pointers are not read): the q8
 * buffer is N * p_pad elements for columns and p * roundup(K, 16) for
 * rows, of 1 byte (INT8, FP8) or 2 (BF16).  INVALID_ARG or UNSUPPORTED
 * as for the decode calls.  Host-only.
 */
bisco_status bisco_layer_sizes(const bisco_layer *L, size_t out_bytes[5]);

/*
 * Scratch bytes bisco_encode needs for an N x K layer (per-column scores and
 * the protected-column map); 0 on invalid sizes.
 */
size_t bisco_encode_workspace_bytes(int32_t N, int32_t K);

/*
 * The same for either protection axis (axis 1: per-row scores, ranks and the
 * protected-row map, 13 bytes per row rounded up); it also covers
 * bisco_encode_with_set.  0 on invalid sizes or axis.
 */
size_t bisco_encode_workspace_bytes_axis(int32_t N, int32_t K, int32_t axis);

/*
 * Offline encoder (Sec. III-E Eq. 8, Eq. 10; Sec. III-C Eq. 3; Sec. III-D
 * Eq. 5-7), deterministic and bit-identical to the fp64 definition:
 *   1. score_j = g_j * sqrt(sum_i W_ij^2) (fp64, ascending i); P = the p
 *      largest, ties to the lower column; stored ascending in prot_idx.
 *   2. per protected column: scale = fp16(max_i |W_ij| / 127),
 *      q8 = clamp(rint_even(W_ij / scale), -127, 127) (0 if scale == 0).
 *   3. stage loop on r = W with protected entries zeroed: n = fp16(||r_c||),
 *      bits = (r_c < 0), r_c -= (+-) n / sqrt(8), protected entries reset
 *      to zero before the next stage.
 * W_bf16: [N][K] device, 16-byte aligned.  g: [K] float device (finite,
 * >= 0) or NULL for g = 1.  L: host struct; its sizes are inputs, its five
 * device buffers outputs (sized by bisco_encoded_sizes).  workspace: device,
 * at least bisco_encode_workspace_bytes(N, K) bytes.  Non-finite weights or
 * an fp16 overflow latch BISCO_ERR_RANGE in the device error word; the
 * outputs are then unspecified.
 * With L->protect_axis = 1 the protected channels are output rows: step 1
 * scores rows, score_i = g_i * sqrt(sum_k W_ik^2) (g: [N], ascending k),
 * step 2 quantises each protected row with one scale (max_k |W_ik| / 127),
 * and step 3 runs on W with the protected rows zeroed.  The workspace is
 * then bisco_encode_workspace_bytes_axis(N, K, 1) bytes.
 */
bisco_status bisco_encode(const uint16_t *W_bf16, const float *g, const bisco_layer *L,
                          void *workspace, size_t workspace_bytes, bisco_stream_t stream);

/*
 * bisco_encode with the protected set given instead of selected: steps 2
 * and 3 above with P = idx_in (device, [p] int32, strictly ascending,
 * columns in [0, K) for axis 0, rows in [0, N) for axis 1; NULL allowed
 * when p == 0), copied to L->prot_idx.  This encodes the three projections
 * of a gated MLP on the one coupled set of bisco_select_coupled (gate and
 * up with axis 1, down with axis 0).  An index out of range or out of order
 * latches BISCO_ERR_INVALID_ARG in the device error word (an out-of-range
 * one is stored as 0; the outputs are then unspecified).  workspace: at
 * least bisco_encode_workspace_bytes_axis(N, K, axis) bytes.
 */
bisco_status bisco_encode_with_set(const uint16_t *W_bf16, const int32_t *idx_in,
                                   const bisco_layer *L, void *workspace, size_t workspace_bytes,
                                   bisco_stream_t stream);

/*
 * Coupled protected set of a gated MLP (Sec. III-E Eq. 9): for intermediate
 * channel j < F,
 *   S_j = gg_j ||Wg[j,:]||_2 + gu_j ||Wu[j,:]||_2 + gd_j ||Wd[:,j]||_2
 * (fp64, each sum of squares in ascending index, the three terms added in
 * that order; a NULL g means 1), and idx_out = the p channels of largest
 * S_j, ties to the lower j, ascending.  Wg, Wu: [F][H] bf16 (gate_proj and
 * up_proj weights), Wd: [H][F] bf16 (down_proj), 16-byte aligned; gg, gu,
 * gd: [F] float or NULL.  F >= 1, H >= 1, 0 <= p <= F.  idx_out: [p] int32
 * device.  workspace: at least bisco_select_coupled_workspace_bytes(F)
 * bytes.  Non-finite weights latch BISCO_ERR_RANGE.
 */
size_t bisco_select_coupled_workspace_bytes(int32_t F);
bisco_status bisco_select_coupled(const uint16_t *Wg_bf16, const uint16_t *Wu_bf16,
                                  const uint16_t *Wd_bf16, const float *gg, const float *gu,
                                  const float *gd, int32_t F, int32_t H, int32_t p,
                                  int32_t *idx_out, void *workspace, size_t workspace_bytes,
                                  bisco_stream_t stream);

/*
 * bisco_encode without a workspace argument, for callers that cannot
 * allocate device memory (for example a host application whose own
 * allocator has reserved the device memory and forbids other cudaMalloc
 * calls, or code that must avoid the device-wide synchronisation that
 * cudaMalloc/cudaFree can cause).  The paper has no counterpart; this is a
 * library convenience.  It calls no cudaMalloc, cudaFree or allocating
 * routine: its scratch is a fixed array inside the library, sized for
 * K <= BISCO_ENCODE_NOALLOC_MAX_K (13 bytes per column, 416 KiB, held on
 * every GPU that loads the library until the process exits).  Larger K
 * returns BISCO_ERR_UNSUPPORTED.  The first call on each device looks up
 * the array's device address (cudaGetSymbolAddress) with that device
 * current; make that first call before any stream capture.  All calls share
 * the one array, so calls that overlap on the GPU race and must be
 * serialised by the caller.  It takes input-column protection with INT8
 * payloads only: protect_axis = 1 or another protect_format returns
 * BISCO_ERR_UNSUPPORTED.  It validates the layer as bisco_encode does
 * (the same BISCO_ERR_INVALID_ARG cases), and its outputs and device
 * errors are those of bisco_encode.
 */
#define BISCO_ENCODE_NOALLOC_MAX_K 32768
bisco_status bisco_encode_noalloc(const uint16_t *W_bf16, const float *g, const bisco_layer *L,
                                  bisco_stream_t stream);

/*
 * Decode-time matrix-vector product for B in [0, 16] activation rows:
 *     y[b][i] = sum_j What[i][j] * x[b][j]        (Sec. III-G Eq. 12, Eq. 10)
 * computed straight from the coded layer (the dense weight is never
 * formed).  x_bf16: [B][K] device bf16 bits; activations are used as fp16,
 * which is exact for 2^-24 <= |x| <= 65504 (larger magnitudes become inf).
 * y: [B][N] float32 device, fully overwritten.  B == 0 is a no-op.
 * The kernel is launched as a programmatic dependent of the previous kernel
 * in the stream: it reads x only after that kernel has completed, but it
 * starts fetching the layer's buffers before, so they must not be written
 * by the kernel immediately ahead of it (bisco_encode ends with an empty
 * kernel for this reason; copies and events order as usual).
 * For a layer with protect_axis = 1, a second kernel then overwrites the
 * protected rows: y[b][prot_idx[t]] = q8_scale[t] * sum_k q8[t][k] * x[b][k]
 * (int8 x bf16 products, exact in fp32, summed in fp32).  The same holds
 * for bisco_gemv_multi and bisco_gemm.
 */
bisco_status bisco_gemv(const bisco_layer *L, const uint16_t *x_bf16, int32_t B, float *y,
                        bisco_stream_t stream);

/*
 * bisco_gemv for G layers that read the same activations, for example the
 * q, k and v projections of one attention layer (Sec. III-G Eq. 12 for each):
 *     y[g][b][i] = sum_j What_g[i][j] * x[b][j]      for g < G
 * in one launch, so the fixed per-launch latency (dependency release,
 * activation staging, reduction tail) is paid once for the group.
 * layers: host array of G structs; all must have the same k_in and stages
 * (n_out and n_protected may differ).  G in [1, BISCO_GEMV_MULTI_MAX].
 * y: host array of G device pointers, y[g] is [B][n_out of layer g] float32,
 * 16-byte aligned, fully overwritten.  x_bf16, B and the launch contract
 * are those of bisco_gemv.  Combinations the grouped kernel does not take
 * (B > 8, K % 128 != 0, shared memory) run as G bisco_gemv launches.
 */
#define BISCO_GEMV_MULTI_MAX 4
bisco_status bisco_gemv_multi(const bisco_layer *layers, int32_t G, const uint16_t *x_bf16,
                              int32_t B, float *const *y, bisco_stream_t stream);

/*
 * A layer's low-rank compensation (Sec. II-D, Sec. III-F), for the fused
 * entry points below: A [rank][K] and Bm [N][rank] bf16 device arrays (the
 * layouts of bisco_lora_apply), 16-byte aligned, and a finite scale.
 * rank 0 means no compensation for that layer (A and Bm are then ignored).
 */
typedef struct bisco_lora {
    const uint16_t *A;
    const uint16_t *Bm;
    int32_t rank;
    float scale;
} bisco_lora;

/*
 * bisco_gemv_multi with each layer's compensation in the same launch:
 *     y[g][i] = sum_j What_g[i][j] * x[j]
 *               + scale_g * sum_r Bm_g[i][r] * sum_k A_g[r][k] * x[k]
 * the quantity bisco_gemv_multi followed by bisco_lora_apply on every
 * layer computes, at batch 1 in one kernel: every CTA forms t = A x for its
 * layer (fp32, summed in a fixed order, so the result does not depend on
 * the launch) and adds Bm t to its rows when it writes them.  loras: host
 * array of G structs.  Taken by the batch-1 row-split kernel only: batch 1,
 * k_in == 4096, stages 1..3, int8 protected columns, every rank a multiple
 * of 8 in [0, BISCO_GEMV_LORA_MAX_RANK]; other combinations return
 * BISCO_ERR_UNSUPPORTED (run bisco_gemv_multi and bisco_lora_apply then).
 * Malformed arguments: BISCO_ERR_INVALID_ARG.  Layers, x and y as for
 * bisco_gemv_multi.  bisco_gemv_lora is the G = 1 case.
 */
#define BISCO_GEMV_LORA_MAX_RANK 64
bisco_status bisco_gemv_multi_lora(const bisco_layer *layers, const bisco_lora *loras, int32_t G,
                                   const uint16_t *x_bf16, float *const *y, bisco_stream_t stream);
bisco_status bisco_gemv_lora(const bisco_layer *L, const bisco_lora *lora, const uint16_t *x_bf16,
                             float *y, bisco_stream_t stream);

/*
 * Prefill matrix product Y[m][i] = sum_j What[i][j] * X[m][j] for any M >= 0
 * (Sec. III-G Eq. 12 with Eq. 10), the same quantity as bisco_gemv.  For
 * M > 16 and K % 128 == 0 it runs on the tcgen05 tensor cores: the decoded
 * weight (fp16, the S stages summed in fp16 -- one rounding of relative
 * size <= 2^-11 per weight for S >= 2) against fp16 activations, fp32
 * accumulation; the protected columns use the int8 values exactly.  Smaller
 * M, or other K, run the decode kernels of bisco_gemv.
 * X_bf16: [M][K] device; Y: [M][N] float32 device, fully overwritten.
 * workspace: device, 16-byte aligned, at least
 * bisco_gemm_workspace_bytes(L, M) bytes (NULL when that is 0).  On the
 * tensor-core path that is the fp16 copy of X, M * (roundup(K,128) +
 * 2 * roundup(p,64)) * 2 bytes (p = 0 for a row-protected layer) rounded up
 * to 256, followed by the partial tiles of the split of the work over the
 * SMs, 160 * 2 * TN * 128 * 4 bytes with TN = 128 for M <= 128 and 256
 * otherwise.  It is overwritten.  Tiles split between SMs are summed by a
 * second kernel in a fixed order, so the result does not depend on timing.
 */
size_t bisco_gemm_workspace_bytes(const bisco_layer *L, int32_t M);
bisco_status bisco_gemm(const bisco_layer *L, const uint16_t *X_bf16, int32_t M, float *Y,
                        void *workspace, size_t workspace_bytes, bisco_stream_t stream);

/*
 * The coded layer decoded to a dense row-major matrix (Sec. III-G Eq. 12
 * with the Eq. 10 overwrite), the materialise-then-multiply alternative to
 * the fused kernels:
 *     out[i][j] = sum_s (bit ? -1 : +1) * n16_{s,i,j/8} / sqrt(8)   j not protected
 *     out[i][j] = scale_j * q8[i][j]                                 j protected
 * The stage sum is formed in fp32 and rounded once after the 1/sqrt(8)
 * scale (to fp32, or from there to bf16 / fp16 with round-to-nearest-even);
 * the protected values are exact in fp32.  With protect_axis = 1 the
 * protected rows are out[prot_idx[t]][k] = q8_scale[t] * q8[t][k].
 * out: [N][K] device, 16-byte aligned, fully overwritten; dtype one of
 * BISCO_DENSE_*.  Asynchronous on `stream` (two kernels).
 */
#define BISCO_DENSE_F32 0
#define BISCO_DENSE_BF16 1
#define BISCO_DENSE_F16 2
bisco_status bisco_decode_dense(const bisco_layer *L, void *out, int32_t dtype,
                                bisco_stream_t stream);

/*
 * One stage of the dense decode (Sec. III-G Eq. 12 term by term), for the
 * sequential residual decode that the packed decode of bisco_decode_dense
 * replaces (Sec. III-G, batched parallel residual decoding):
 *     out[i][j]  = (bit_{stage,i,j} ? -1 : +1) * n16_{stage,i,j/8} / sqrt(8)   accumulate == 0
 *     out[i][j] += the same                                                    accumulate != 0
 * for every column, each term rounded once to fp32.  When stage is the last
 * one (S - 1) the protected columns (rows, protect_axis = 1) are then
 * overwritten as in bisco_decode_dense, so calling stages 0 .. S-1 in order
 * with accumulate = (stage > 0) yields What, the stage terms added in stage
 * order.  out: [N][K] fp32 device, 16-byte aligned.  stage outside
 * [0, S) returns BISCO_ERR_INVALID_ARG.  Asynchronous on `stream`.
 */
bisco_status bisco_decode_dense_stage(const bisco_layer *L, int32_t stage, float *out,
                                      int32_t accumulate, bisco_stream_t stream);

/*
 * The learned decoder step (Sec. III-A Eq. 1; the decoder ablation compares
 * a symmetric, sign-symmetric decoder with a linear one).  A stage's chunk
 * decodes to n16 * D_s(q); with b = 8 the code q takes 256 values, so D_s is
 * passed as its table:
 *   tables [S][256][8] uint16, binary16 bits, device, 16-byte aligned;
 *   tables[s][v][k] = D_s(q(v))_k, with bit k of v set <=> q_k < 0.
 * The identity decoder is (bit k of v ? -1 : +1) / sqrt(8) (rounded to
 * binary16); a linear decoder A_s q and the perceptron of the ablation are
 * evaluated by the caller into the same form.  The decoded weight is
 *   What[i][8c + k] = sum_s n16_{s,i,c} * tables[s][code_{s,i,c}][k]
 * (fp16 x fp16 products, exact in fp32, summed in fp32), with the protected
 * columns (or rows, protect_axis = 1) as for bisco_gemv.
 * bisco_gemv_table: y[b][i] = sum_j What[i][j] * x[b][j] for B in [0, 16],
 * one warp per output row (not tuned for bandwidth), fp32 throughout.
 * bisco_decode_dense_table: What as a dense [N][K] fp32 / bf16 / fp16
 * matrix (BISCO_DENSE_*), rounded once from fp32.
 * Arguments and errors are otherwise those of bisco_gemv and
 * bisco_decode_dense; protected columns need the INT8 payload
 * (BISCO_ERR_UNSUPPORTED otherwise), protected rows take any format.
 */
bisco_status bisco_gemv_table(const bisco_layer *L, const uint16_t *tables, const uint16_t *x_bf16,
                              int32_t B, float *y, bisco_stream_t stream);
bisco_status bisco_decode_dense_table(const bisco_layer *L, const uint16_t *tables, void *out,
                                      int32_t dtype, bisco_stream_t stream);

/*
 * Low-rank compensation (the optional LoRA path of Sec. II-D and Sec. III-F:
 * adapters trained after the codes are fixed, kept apart from the coded
 * layer's storage), added to an output the layer has already written:
 *     t[b][r]  = sum_k A[r][k] * x[b][k]                (fp32 accumulation)
 *     y[b][n] += scale * sum_r Bm[n][r] * t[b][r]        (fp32)
 * A: [rank][K] bf16 and Bm: [N][rank] bf16 (the layouts of a PyTorch
 * lora_A / lora_B weight); x_bf16: [batch][K]; y: [batch][N] float32, read
 * and written (call it after bisco_gemv / bisco_gemm on the same stream);
 * t: [batch][rank] float32 scratch, overwritten.  K >= 8, K % 8 == 0,
 * N >= 1, 8 <= rank <= BISCO_LORA_MAX_RANK with rank % 8 == 0,
 * 1 <= batch <= 65535, scale finite; else BISCO_ERR_INVALID_ARG.  Every
 * pointer 16-byte aligned.  Asynchronous on `stream` (two kernels); the
 * result does not depend on the launch (fixed summation order).
 */
#define BISCO_LORA_MAX_RANK 256
bisco_status bisco_lora_apply(const uint16_t *A, const uint16_t *Bm, int32_t rank, int32_t N,
                              int32_t K, float scale, const uint16_t *x_bf16, int32_t batch,
                              float *y, float *t, bisco_stream_t stream);

/*
 * A protected-column index outside [0, K) (or a list that is not ascending)
 * found by a kernel is skipped and latches BISCO_ERR_INVALID_ARG in the
 * device error word.
 *
 * Synchronises `stream`, returns the device error word of the current device
 * (BISCO_OK if clear) and clears it.  BISCO_ERR_CUDA if the synchronisation
 * itself fails.
 */
bisco_status bisco_get_device_error(bisco_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* BISCO_H */
