// fxpq_conv_tc_scale.cu -- the tensor-core C-Block kernels of layers with a Scale layer (a BN layer
// rewritten as aleph1 * A + aleph2, Sec. IV-A.1): the same contraction as fxpq_conv_tc.cu, with the
// per-channel multiply and aligned add in the epilogue before ReLU and the FxP-QLayer.
#include "fxpq_conv_tc.cuh"

namespace fxpq {

using namespace tc;

namespace {

std::mutex g_sc_mu;
bool g_sc_attr_set = false;

}  // namespace

fxpq_status launch_conv_tc_scaled(const TcParams& P, int BN, bool acc64, int grid, cudaStream_t st) {
    {
        std::lock_guard<std::mutex> lk(g_sc_mu);
        if (!g_sc_attr_set) {
            if (cudaFuncSetAttribute(conv_tc_kernel<64, long long, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<64>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<64, int, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<64>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<128, int, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<128>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<256, int, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<256>()) != cudaSuccess)
                return FXPQ_ERR_CUDA;
            g_sc_attr_set = true;
        }
    }
    if (acc64)
        conv_tc_kernel<64, long long, true><<<grid, tc_threads(64), tc_smem_bytes<64>(), st>>>(P);
    else if (BN == 64)
        conv_tc_kernel<64, int, true><<<grid, tc_threads(64), tc_smem_bytes<64>(), st>>>(P);
    else if (BN == 128)
        conv_tc_kernel<128, int, true><<<grid, tc_threads(128), tc_smem_bytes<128>(), st>>>(P);
    else
        conv_tc_kernel<256, int, true><<<grid, tc_threads(256), tc_smem_bytes<256>(), st>>>(P);
    return after_launch("conv_tc_scale");
}

}  // namespace fxpq
