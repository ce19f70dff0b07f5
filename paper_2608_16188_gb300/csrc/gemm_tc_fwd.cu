// gemm_tc_fwd.cu -- tensor-map encoding and the forward launches of the
// tcgen05 grouped GEMM:
//   FC1 + GELU: H = Xe W1, A = GELU(H)   (A: Xe K-major; B: W1 [d,f] MN-major)
//   FC2:        Ye = A W2                (A: A  K-major; B: W2 [f,d] MN-major)
#include "gemm_tc2.cuh"

namespace vmoe {
namespace tc {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encoder() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

bool make_map(CUtensorMap *map, const void *base, uint64_t inner, uint64_t mid, uint64_t outer,
              uint32_t box_mid, uint64_t outer_stride_elems) {
    EncodeTiledFn fn = encoder();
    if (!fn) return false;
    cuuint64_t dims[3] = {inner, mid, outer};
    cuuint64_t strides[2] = {inner * 2, (outer_stride_elems ? outer_stride_elems : inner * mid) * 2};
    cuuint32_t box[3] = {64, box_mid, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_map_chunked(CUtensorMap *map, const void *base, uint64_t mn, uint64_t rows,
                      uint64_t outer, uint32_t box_rows, uint32_t box_chunks,
                      uint64_t outer_stride_elems) {
    EncodeTiledFn fn = encoder();
    if (!fn || mn % 64 != 0) return false;
    cuuint64_t dims[4] = {64, rows, mn / 64, outer};
    // bytes: row, chunk, group
    cuuint64_t strides[3] = {mn * 2, 128, (outer_stride_elems ? outer_stride_elems : rows * mn) * 2};
    cuuint32_t box[4] = {64, box_rows, box_chunks, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace tc

using namespace tc;

int launch_expert_fwd_bf16(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *w1,
                           const __nv_bfloat16 *w2, const int32_t *load, __nv_bfloat16 *h,
                           __nv_bfloat16 *act, __nv_bfloat16 *ye, cudaStream_t s) {
    int st = row_gemm<EPI_GELU, true>(p, xe, p.d, w1, p.f, load, h, act, nullptr, s, "tc_fc1_gelu");
    if (st != VMOE_OK) return st;
    return row_gemm<EPI_STORE, true>(p, act, p.f, w2, p.d, load, ye, nullptr, nullptr, s, "tc_fc2");
}

// Attention experts, forward: QKV = Xe W_qkv, the attention core (O and the
// row log-sum-exp, attention.cu), Ye = O W_o.
int launch_attn_expert_fwd(const Dims &p, int H, const __nv_bfloat16 *xe, const __nv_bfloat16 *wqkv,
                           const __nv_bfloat16 *wo, const int32_t *load, __nv_bfloat16 *qkv,
                           __nv_bfloat16 *o, float *lse, __nv_bfloat16 *ye, cudaStream_t s) {
    const int hd = H * 64;
    int st = row_gemm<EPI_STORE, true>(p, xe, p.d, wqkv, 3 * hd, load, qkv, nullptr, nullptr, s, "attn_qkv");
    if (st != VMOE_OK) return st;
    if ((st = launch_attn_core_fwd(p.G(), p.C, H, load, qkv, o, lse, s)) != VMOE_OK) return st;
    return row_gemm<EPI_STORE, true>(p, o, hd, wo, p.d, load, ye, nullptr, nullptr, s, "attn_out");
}

}  // namespace vmoe
