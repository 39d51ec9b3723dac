// api.cu -- the extern "C" entry points declared in include/bisco.h:
// argument validation, the per-device error word, tensor-map encoding and
// dispatch to the kernels in encode.cu / gemv.cu / gemm.cu.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdint.h>

#include <cmath>
#include <mutex>

#include "bisco_host.h"

namespace bisco {

__device__ int g_device_error;

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int *g_err_ptr[kMaxDevices] = {};
int g_sms[kMaxDevices] = {};
PFN_cuTensorMapEncodeTiled_v12000 g_encode_tiled = nullptr;

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int current_device() {
    int d = -1;
    if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
    return d;
}


// Layers whose protected set the decode kernels do not take themselves:
// output rows (rows.cu) and payloads other than INT8 (formats.cu) -- except
// at batch 1, where the row-split kernel takes protected columns and rows in
// every payload format.
bool needs_epilogue(const bisco_layer &L) {
    return L.n_protected > 0 &&
           (L.protect_axis == 1 || L.protect_format != BISCO_PROT_INT8);
}

// The binary spherical stages of such a layer alone: the decode kernels run
// on this copy (no protected set; they read none of the protected buffers
// when p == 0), then epilogue() applies the protected set.
bisco_layer bsq_only(const bisco_layer &L) {
    bisco_layer b = L;
    b.n_protected = 0;
    b.protect_axis = 0;
    b.protect_format = BISCO_PROT_INT8;
    return b;
}

bisco_status epilogue(const bisco_layer &L, const uint16_t *X, int M, float *Y, int *err,
                      cudaStream_t s) {
    if (L.protect_axis == 1) return launch_rows_apply(L, X, M, Y, err, s);
    return launch_prot_fix(L, X, M, Y, err, s);
}

bisco_status dense_epilogue(const bisco_layer &L, void *out, int dtype, int *err, cudaStream_t s) {
    if (L.protect_axis == 1) return launch_rows_dense(L, out, dtype, err, s);
    return launch_dense_fmt(L, out, dtype, err, s);
}

}  // namespace

// Validates the sizes of a layer; buffers too when check_buffers.
bisco_status check_layer(const bisco_layer *L, bool check_buffers) {
    if (!L) return BISCO_ERR_INVALID_ARG;
    if (L->n_out < 1 || L->k_in < 8 || L->k_in % 8 != 0) return BISCO_ERR_INVALID_ARG;
    if (L->stages < 1 || L->stages > 3) return BISCO_ERR_INVALID_ARG;
    if (L->protect_axis != 0 && L->protect_axis != 1) return BISCO_ERR_INVALID_ARG;
    const int32_t p_max = L->protect_axis == 1 ? L->n_out : L->k_in;
    if (L->n_protected < 0 || L->n_protected > p_max) return BISCO_ERR_INVALID_ARG;
    if (L->protect_format < BISCO_PROT_INT8 || L->protect_format > BISCO_PROT_BF16)
        return BISCO_ERR_INVALID_ARG;
    if (L->chunk_dim != 8) return BISCO_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(L->n_out) * L->k_in > (int64_t(1) << 40)) return BISCO_ERR_INVALID_ARG;
    if (!check_buffers) return BISCO_OK;
    if (!L->codes || !L->norms || !aligned16(L->codes) || !aligned16(L->norms))
        return BISCO_ERR_INVALID_ARG;
    if (L->n_protected > 0) {
        if (!L->q8 || !L->q8_scale || !L->prot_idx) return BISCO_ERR_INVALID_ARG;
        if (!aligned16(L->q8) || !aligned16(L->q8_scale) || !aligned16(L->prot_idx))
            return BISCO_ERR_INVALID_ARG;
    }
    return BISCO_OK;
}

int *device_error_word(bisco_status *st) {
    const int d = current_device();
    if (d < 0) {
        *st = BISCO_ERR_CUDA;
        return nullptr;
    }
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_err_ptr[d]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) {
            *st = BISCO_ERR_CUDA;
            return nullptr;
        }
        g_err_ptr[d] = static_cast<int *>(p);
    }
    *st = BISCO_OK;
    return g_err_ptr[d];
}

int num_sms() {
    const int d = current_device();
    if (d < 0) return 148;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_sms[d]) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, d) != cudaSuccess || v <= 0)
            v = 148;
        g_sms[d] = v;
    }
    return g_sms[d];
}

bool encode_tensor_map(CUtensorMap *map, CUtensorMapDataType dtype, int rank, void *base,
                       const uint64_t *dims, const uint64_t *strides_bytes, const uint32_t *box,
                       CUtensorMapSwizzle swizzle) {
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_encode_tiled) {
            cudaDriverEntryPointQueryResult q;
            void *fn = nullptr;
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                 cudaEnableDefault, &q) != cudaSuccess ||
                q != cudaDriverEntryPointSuccess || !fn)
                return false;
            g_encode_tiled = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
        }
    }
    cuuint64_t gdim[5], gstr[4];
    cuuint32_t bdim[5], estr[5];
    for (int i = 0; i < rank; ++i) {
        gdim[i] = dims[i];
        bdim[i] = box[i];
        estr[i] = 1;
        if (i + 1 < rank) gstr[i] = strides_bytes[i];
    }
    const CUresult r = g_encode_tiled(map, dtype, static_cast<cuuint32_t>(rank), base, gdim, gstr,
                                      bdim, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace bisco

using namespace bisco;

extern "C" {

int32_t bisco_abi_version(void) { return BISCO_ABI_VERSION; }

const char *bisco_status_string(int32_t status) {
    switch (status) {
        case BISCO_OK: return "ok";
        case BISCO_ERR_INVALID_ARG: return "invalid argument";
        case BISCO_ERR_UNSUPPORTED: return "unsupported configuration";
        case BISCO_ERR_RANGE: return "value out of range (non-finite weight or fp16 overflow)";
        case BISCO_ERR_CUDA: return "CUDA runtime error";
        case BISCO_ERR_TIMEOUT: return "bounded device wait expired";
        default: return "unknown status";
    }
}

bisco_status bisco_encoded_sizes(int32_t N, int32_t K, int32_t d, int32_t S, int32_t p,
                                 size_t out_bytes[5]) {
    if (!out_bytes) return BISCO_ERR_INVALID_ARG;
    if (N < 1 || K < 8 || K % 8 != 0 || S < 1 || S > 3 || p < 0 || p > K)
        return BISCO_ERR_INVALID_ARG;
    if (d != 8) return BISCO_ERR_UNSUPPORTED;
    const size_t C = static_cast<size_t>(K) / 8;
    const size_t p_pad = (static_cast<size_t>(p) + 15) / 16 * 16;
    out_bytes[0] = static_cast<size_t>(S) * N * C;
    out_bytes[1] = static_cast<size_t>(S) * N * C * 2;
    out_bytes[2] = static_cast<size_t>(N) * p_pad;
    out_bytes[3] = static_cast<size_t>(p) * 2;
    out_bytes[4] = static_cast<size_t>(p) * 4;
    return BISCO_OK;
}

bisco_status bisco_layer_sizes(const bisco_layer *L, size_t out_bytes[5]) {
    if (!out_bytes) return BISCO_ERR_INVALID_ARG;
    const bisco_status st = check_layer(L, false);
    if (st != BISCO_OK) return st;
    const size_t N = static_cast<size_t>(L->n_out), K = static_cast<size_t>(L->k_in);
    const size_t S = static_cast<size_t>(L->stages), p = static_cast<size_t>(L->n_protected);
    const size_t C = K / 8;
    out_bytes[0] = S * N * C;
    out_bytes[1] = S * N * C * 2;
    const size_t elem = L->protect_format == BISCO_PROT_BF16 ? 2 : 1;
    if (L->protect_axis == 1)
        out_bytes[2] = p * ((K + 15) / 16 * 16) * elem;
    else
        out_bytes[2] = N * ((p + 15) / 16 * 16) * elem;
    out_bytes[3] = p * 2;
    out_bytes[4] = p * 4;
    return BISCO_OK;
}

size_t bisco_encode_workspace_bytes(int32_t N, int32_t K) { return encode_workspace_bytes(N, K); }

size_t bisco_encode_workspace_bytes_axis(int32_t N, int32_t K, int32_t axis) {
    return encode_workspace_bytes_axis(N, K, axis);
}

size_t bisco_select_coupled_workspace_bytes(int32_t F) { return select_coupled_workspace_bytes(F); }

bisco_status bisco_encode(const uint16_t *W_bf16, const float *g, const bisco_layer *L,
                          void *workspace, size_t workspace_bytes, bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (!W_bf16 || !aligned16(W_bf16) || (g && (reinterpret_cast<uintptr_t>(g) & 3u)))
        return BISCO_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) ||
        workspace_bytes < encode_workspace_bytes_axis(L->n_out, L->k_in, L->protect_axis))
        return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    if (L->protect_axis == 1)
        return launch_encode_rows(W_bf16, g, *L, workspace, err,
                                  reinterpret_cast<cudaStream_t>(stream));
    return launch_encode(W_bf16, g, *L, workspace, err, reinterpret_cast<cudaStream_t>(stream));
}

bisco_status bisco_encode_with_set(const uint16_t *W_bf16, const int32_t *idx_in,
                                   const bisco_layer *L, void *workspace, size_t workspace_bytes,
                                   bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (!W_bf16 || !aligned16(W_bf16)) return BISCO_ERR_INVALID_ARG;
    if (L->n_protected > 0 && (!idx_in || (reinterpret_cast<uintptr_t>(idx_in) & 3u)))
        return BISCO_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) ||
        workspace_bytes < encode_workspace_bytes_axis(L->n_out, L->k_in, L->protect_axis))
        return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    return launch_encode_with_set(W_bf16, idx_in, *L, workspace, err,
                                  reinterpret_cast<cudaStream_t>(stream));
}

bisco_status bisco_select_coupled(const uint16_t *Wg_bf16, const uint16_t *Wu_bf16,
                                  const uint16_t *Wd_bf16, const float *gg, const float *gu,
                                  const float *gd, int32_t F, int32_t H, int32_t p,
                                  int32_t *idx_out, void *workspace, size_t workspace_bytes,
                                  bisco_stream_t stream) {
    if (F < 1 || H < 1 || p < 0 || p > F) return BISCO_ERR_INVALID_ARG;
    if (static_cast<int64_t>(F) * H > (int64_t(1) << 40)) return BISCO_ERR_INVALID_ARG;
    const void *w[3] = {Wg_bf16, Wu_bf16, Wd_bf16};
    for (const void *q : w)
        if (!q || !aligned16(q)) return BISCO_ERR_INVALID_ARG;
    const float *g[3] = {gg, gu, gd};
    for (const float *q : g)
        if (q && (reinterpret_cast<uintptr_t>(q) & 3u)) return BISCO_ERR_INVALID_ARG;
    if (p > 0 && (!idx_out || (reinterpret_cast<uintptr_t>(idx_out) & 3u)))
        return BISCO_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) ||
        workspace_bytes < select_coupled_workspace_bytes(F))
        return BISCO_ERR_INVALID_ARG;
    bisco_status st;
    int *err = device_error_word(&st);
    if (!err) return st;
    return launch_select_coupled(Wg_bf16, Wu_bf16, Wd_bf16, gg, gu, gd, F, H, p, idx_out,
                                 workspace, err, reinterpret_cast<cudaStream_t>(stream));
}

bisco_status bisco_gemv(const bisco_layer *L, const uint16_t *x_bf16, int32_t B, float *y,
                        bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (B < 0 || B > 16) return BISCO_ERR_INVALID_ARG;
    if (B == 0) return BISCO_OK;
    if (!x_bf16 || !y || !aligned16(x_bf16) || !aligned16(y)) return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (needs_epilogue(*L)) {
        // batch 1, protected columns in an FP8 / bf16 payload or protected
        // rows: the batch-1 kernel takes those itself, in one launch
        if (B == 1 && !getenv("BISCO_GEMV_MODE")) {
            bool launched = false;
            st = launch_gemv_b1(L, 1, x_bf16, &y, err, s, &launched);
            if (launched || st != BISCO_OK) return st;
        }
        st = launch_gemv(bsq_only(*L), x_bf16, B, y, err, s);
        if (st != BISCO_OK) return st;
        return epilogue(*L, x_bf16, B, y, err, s);
    }
    return launch_gemv(*L, x_bf16, B, y, err, s);
}

bisco_status bisco_gemv_multi(const bisco_layer *layers, int32_t G, const uint16_t *x_bf16,
                              int32_t B, float *const *y, bisco_stream_t stream) {
    if (!layers || !y || G < 1 || G > BISCO_GEMV_MULTI_MAX) return BISCO_ERR_INVALID_ARG;
    for (int g = 0; g < G; ++g) {
        const bisco_status st = check_layer(&layers[g], true);
        if (st != BISCO_OK) return st;
        if (layers[g].k_in != layers[0].k_in || layers[g].stages != layers[0].stages)
            return BISCO_ERR_INVALID_ARG;
    }
    if (B < 0 || B > 16) return BISCO_ERR_INVALID_ARG;
    if (B == 0) return BISCO_OK;
    if (!x_bf16 || !aligned16(x_bf16)) return BISCO_ERR_INVALID_ARG;
    for (int g = 0; g < G; ++g)
        if (!y[g] || !aligned16(y[g])) return BISCO_ERR_INVALID_ARG;
    bisco_status st;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    bisco_layer stages[BISCO_GEMV_MULTI_MAX];
    bool any = false;
    for (int g = 0; g < G; ++g) {
        const bool e = needs_epilogue(layers[g]);
        any |= e;
        stages[g] = e ? bsq_only(layers[g]) : layers[g];
    }
    if (!any) return launch_gemv_multi(layers, G, x_bf16, B, y, err, s);
    // batch 1, protected columns or rows in any payload format: one launch
    // of the batch-1 kernel
    if (B == 1 && !getenv("BISCO_GEMV_MODE")) {
        bool launched = false;
        st = launch_gemv_b1(layers, G, x_bf16, y, err, s, &launched);
        if (launched || st != BISCO_OK) return st;
    }
    st = launch_gemv_multi(stages, G, x_bf16, B, y, err, s);
    for (int g = 0; g < G && st == BISCO_OK; ++g)
        if (needs_epilogue(layers[g])) st = epilogue(layers[g], x_bf16, B, y[g], err, s);
    return st;
}

bisco_status bisco_gemv_multi_lora(const bisco_layer *layers, const bisco_lora *loras, int32_t G,
                                   const uint16_t *x_bf16, float *const *y, bisco_stream_t stream) {
    if (!layers || !loras || !y || G < 1 || G > BISCO_GEMV_MULTI_MAX) return BISCO_ERR_INVALID_ARG;
    if (!x_bf16 || !aligned16(x_bf16)) return BISCO_ERR_INVALID_ARG;
    for (int g = 0; g < G; ++g) {
        const bisco_status st = check_layer(&layers[g], true);
        if (st != BISCO_OK) return st;
        if (layers[g].k_in != layers[0].k_in || layers[g].stages != layers[0].stages)
            return BISCO_ERR_INVALID_ARG;
        if (!y[g] || !aligned16(y[g])) return BISCO_ERR_INVALID_ARG;
        const bisco_lora &r = loras[g];
        if (r.rank < 0 || r.rank > BISCO_GEMV_LORA_MAX_RANK || r.rank % 8 != 0) return BISCO_ERR_INVALID_ARG;
        if (r.rank > 0 && (!r.A || !r.Bm || !aligned16(r.A) || !aligned16(r.Bm) || !std::isfinite(r.scale)))
            return BISCO_ERR_INVALID_ARG;
        if (needs_epilogue(layers[g])) return BISCO_ERR_UNSUPPORTED;   // int8 columns only
    }
    if (layers[0].k_in != 4096) return BISCO_ERR_UNSUPPORTED;
    bisco_status st;
    int *err = device_error_word(&st);
    if (!err) return st;
    bool launched = false;
    st = launch_gemv_b1(layers, G, x_bf16, y, err, reinterpret_cast<cudaStream_t>(stream), &launched, loras);
    if (st != BISCO_OK) return st;
    return launched ? BISCO_OK : BISCO_ERR_UNSUPPORTED;
}

bisco_status bisco_gemv_lora(const bisco_layer *L, const bisco_lora *lora, const uint16_t *x_bf16,
                             float *y, bisco_stream_t stream) {
    if (!L || !lora || !y) return BISCO_ERR_INVALID_ARG;
    return bisco_gemv_multi_lora(L, lora, 1, x_bf16, &y, stream);
}

size_t bisco_gemm_workspace_bytes(const bisco_layer *L, int32_t M) {
    if (M < 0 || check_layer(L, false) != BISCO_OK) return 0;
    return gemm_workspace_bytes(needs_epilogue(*L) ? bsq_only(*L) : *L, M);
}

bisco_status bisco_gemm(const bisco_layer *L, const uint16_t *X_bf16, int32_t M, float *Y,
                        void *workspace, size_t workspace_bytes, bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (M < 0) return BISCO_ERR_INVALID_ARG;
    if (M == 0) return BISCO_OK;
    if (!X_bf16 || !Y || !aligned16(X_bf16) || !aligned16(Y)) return BISCO_ERR_INVALID_ARG;
    const bisco_layer Ls = needs_epilogue(*L) ? bsq_only(*L) : *L;
    const size_t need = gemm_workspace_bytes(Ls, M);
    if (need && (!workspace || !aligned16(workspace) || workspace_bytes < need))
        return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    st = launch_gemm(Ls, X_bf16, M, Y, workspace, workspace_bytes, err, s);
    if (st != BISCO_OK || !needs_epilogue(*L)) return st;
    return epilogue(*L, X_bf16, M, Y, err, s);
}

bisco_status bisco_decode_dense(const bisco_layer *L, void *out, int32_t dtype,
                                bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (dtype != BISCO_DENSE_F32 && dtype != BISCO_DENSE_BF16 && dtype != BISCO_DENSE_F16)
        return BISCO_ERR_INVALID_ARG;
    if (!out || !aligned16(out)) return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (needs_epilogue(*L)) {
        st = launch_decode_dense(bsq_only(*L), out, dtype, err, s);
        if (st != BISCO_OK) return st;
        return dense_epilogue(*L, out, dtype, err, s);
    }
    return launch_decode_dense(*L, out, dtype, err, s);
}

bisco_status bisco_decode_dense_stage(const bisco_layer *L, int32_t stage, float *out,
                                      int32_t accumulate, bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (stage < 0 || stage >= L->stages) return BISCO_ERR_INVALID_ARG;
    if (!out || !aligned16(out)) return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    st = launch_decode_stage(*L, stage, out, accumulate != 0, s);
    if (st != BISCO_OK || stage != L->stages - 1 || L->n_protected == 0) return st;
    // after the last stage the protected set overwrites its columns (or rows)
    if (needs_epilogue(*L)) return dense_epilogue(*L, out, BISCO_DENSE_F32, err, s);
    return launch_dense_protected_f32(*L, out, err, s);
}

bisco_status bisco_gemv_table(const bisco_layer *L, const uint16_t *tables, const uint16_t *x_bf16,
                              int32_t B, float *y, bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    // a column payload other than INT8 is corrected against the identity
    // decoder's stage value (formats.cu), not a table's: rows only
    if (L->protect_format != BISCO_PROT_INT8 && L->protect_axis == 0) return BISCO_ERR_UNSUPPORTED;
    if (B < 0 || B > 16) return BISCO_ERR_INVALID_ARG;
    if (!tables || !aligned16(tables)) return BISCO_ERR_INVALID_ARG;
    if (B == 0) return BISCO_OK;
    if (!x_bf16 || !y || !aligned16(x_bf16) || !aligned16(y)) return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // batch 1, K a multiple of 4096: the row-split kernel in table mode
    if (B == 1 && L->protect_axis == 0 && !getenv("BISCO_GEMV_MODE")) {
        bool launched = false;
        st = launch_gemv_b1(L, 1, x_bf16, &y, err, s, &launched, nullptr, tables);
        if (launched || st != BISCO_OK) return st;
    }
    if (L->protect_axis == 1) {
        st = launch_gemv_table(bsq_only(*L), tables, x_bf16, B, y, err, s);
        if (st != BISCO_OK) return st;
        return launch_rows_apply(*L, x_bf16, B, y, err, s);
    }
    return launch_gemv_table(*L, tables, x_bf16, B, y, err, s);
}

bisco_status bisco_decode_dense_table(const bisco_layer *L, const uint16_t *tables, void *out,
                                      int32_t dtype, bisco_stream_t stream) {
    bisco_status st = check_layer(L, true);
    if (st != BISCO_OK) return st;
    if (L->protect_format != BISCO_PROT_INT8 && L->protect_axis == 0) return BISCO_ERR_UNSUPPORTED;
    if (dtype != BISCO_DENSE_F32 && dtype != BISCO_DENSE_BF16 && dtype != BISCO_DENSE_F16)
        return BISCO_ERR_INVALID_ARG;
    if (!tables || !aligned16(tables) || !out || !aligned16(out)) return BISCO_ERR_INVALID_ARG;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (L->protect_axis == 1) {
        st = launch_dense_table(bsq_only(*L), tables, out, dtype, err, s);
        if (st != BISCO_OK) return st;
        return launch_rows_dense(*L, out, dtype, err, s);
    }
    return launch_dense_table(*L, tables, out, dtype, err, s);
}

bisco_status bisco_lora_apply(const uint16_t *A, const uint16_t *Bm, int32_t rank, int32_t N,
                              int32_t K, float scale, const uint16_t *x_bf16, int32_t batch,
                              float *y, float *t, bisco_stream_t stream) {
    if (rank < 8 || rank > BISCO_LORA_MAX_RANK || rank % 8 != 0) return BISCO_ERR_INVALID_ARG;
    if (N < 1 || K < 8 || K % 8 != 0 || batch < 1 || batch > 65535) return BISCO_ERR_INVALID_ARG;
    if (!std::isfinite(scale)) return BISCO_ERR_INVALID_ARG;
    const void *ptrs[5] = {A, Bm, x_bf16, y, t};
    for (const void *q : ptrs)
        if (!q || !aligned16(q)) return BISCO_ERR_INVALID_ARG;
    return launch_lora_apply(A, Bm, rank, N, K, scale, x_bf16, batch, y, t,
                             reinterpret_cast<cudaStream_t>(stream));
}

bisco_status bisco_get_device_error(bisco_stream_t stream) {
    bisco_status st;
    int *err = device_error_word(&st);
    if (!err) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return BISCO_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, err, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return BISCO_ERR_CUDA;
    if (v != 0 && cudaMemset(err, 0, sizeof v) != cudaSuccess) return BISCO_ERR_CUDA;
    return static_cast<bisco_status>(v);
}

}  // extern "C"
