// bisco_host.h -- host-side declarations shared by the library's
// translation units (not part of the public ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/bisco.h"

namespace bisco {

// Validates the sizes of a layer (api.cu); its buffers too when
// check_buffers.
bisco_status check_layer(const bisco_layer *L, bool check_buffers);

// Device error word of the current device (set up on first use).
int *device_error_word(bisco_status *st);

// cuTensorMapEncodeTiled through the runtime's driver entry point.
bool encode_tensor_map(CUtensorMap *map, CUtensorMapDataType dtype, int rank, void *base,
                       const uint64_t *dims, const uint64_t *strides_bytes, const uint32_t *box,
                       CUtensorMapSwizzle swizzle);

int num_sms();

size_t encode_workspace_bytes(int N, int K);
bisco_status launch_encode(const uint16_t *W, const float *g, const bisco_layer &L,
                           void *workspace, int *err, cudaStream_t stream);
bisco_status launch_gemv(const bisco_layer &L, const uint16_t *x, int B, float *y, int *err,
                         cudaStream_t stream);
bisco_status launch_gemv_multi(const bisco_layer *Ls, int G, const uint16_t *x, int B,
                               float *const *y, int *err, cudaStream_t stream);
// Batch-1 decode for G <= 4 layers sharing x with K % 4096 == 0 and column
// protection in any payload format (gemv_b1.cu), with each layer's low-rank
// compensation when loras is not null (K == 4096 only); *launched stays
// false when the layers do not fit its plan.
// With tables (the decoder tables of bisco_gemv_table, [S][256][8] fp16) it
// runs the learned decoder step instead of the sign decode (one layer, int8
// payloads).
bisco_status launch_gemv_b1(const bisco_layer *Ls, int G, const uint16_t *x, float *const *y,
                            int *err, cudaStream_t stream, bool *launched,
                            const bisco_lora *loras = nullptr, const uint16_t *tables = nullptr);
// Output-row protection and the coupled MLP set (encode.cu, rows.cu).
size_t encode_workspace_bytes_axis(int N, int K, int axis);
size_t select_coupled_workspace_bytes(int F);
bisco_status launch_encode_rows(const uint16_t *W, const float *g, const bisco_layer &L,
                                void *workspace, int *err, cudaStream_t stream);
bisco_status launch_encode_with_set(const uint16_t *W, const int32_t *idx_in,
                                    const bisco_layer &L, void *workspace, int *err,
                                    cudaStream_t stream);
bisco_status launch_select_coupled(const uint16_t *Wg, const uint16_t *Wu, const uint16_t *Wd,
                                   const float *gg, const float *gu, const float *gd, int F,
                                   int H, int p, int32_t *idx_out, void *workspace, int *err,
                                   cudaStream_t stream);
bisco_status launch_rows_apply(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                               cudaStream_t stream);
bisco_status launch_rows_dense(const bisco_layer &L, void *out, int dtype, int *err,
                               cudaStream_t stream);
// Protected payloads other than INT8 (formats.cu): the encoder's
// quantiser, the correction after the stage-only decode kernels, and the
// dense overwrite.
bisco_status launch_q_fmt(const uint16_t *W, const bisco_layer &L, int *err, cudaStream_t stream);
bisco_status launch_q_fmt_rows(const uint16_t *W, const bisco_layer &L, int *err,
                               cudaStream_t stream);
bisco_status launch_prot_fix(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                             cudaStream_t stream);
bisco_status launch_dense_fmt(const bisco_layer &L, void *out, int dtype, int *err,
                              cudaStream_t stream);
// The learned decoder step in table form (decoder.cu).
bisco_status launch_gemv_table(const bisco_layer &L, const uint16_t *tables, const uint16_t *x,
                               int B, float *y, int *err, cudaStream_t stream);
bisco_status launch_dense_table(const bisco_layer &L, const uint16_t *tables, void *out, int dtype,
                                int *err, cudaStream_t stream);
size_t gemm_workspace_bytes(const bisco_layer &L, int M);
bisco_status launch_gemm(const bisco_layer &L, const uint16_t *X, int M, float *Y,
                         void *workspace, size_t ws_bytes, int *err, cudaStream_t stream);
bisco_status launch_decode_dense(const bisco_layer &L, void *out, int dtype, int *err,
                                 cudaStream_t stream);
// One stage into a dense fp32 matrix, and the INT8 protected-column
// overwrite of that matrix (dense.cu).
bisco_status launch_decode_stage(const bisco_layer &L, int stage, float *out, bool accumulate,
                                 cudaStream_t stream);
bisco_status launch_dense_protected_f32(const bisco_layer &L, float *out, int *err, cudaStream_t stream);

// bisco_lora_apply's two kernels (arguments already validated).
bisco_status launch_lora_apply(const uint16_t *A, const uint16_t *Bm, int rank, int N, int K,
                               float scale, const uint16_t *x, int batch, float *y, float *t,
                               cudaStream_t stream);

}  // namespace bisco
