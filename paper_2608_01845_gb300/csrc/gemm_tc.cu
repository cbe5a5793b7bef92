// tcgen05 GEMM (placeholder until the TMEM kernel lands).
#include "dit_kernels.cuh"
namespace wdc {
bool tc_gemm_supported(int, int, int) { return false; }
wdc_status tc_gemm(Ctx* c, const void*, const void*, int, int, int, const Epi&, cudaStream_t) {
    return fail(c, WDC_ERR_UNSUPPORTED, "tcgen05 GEMM not built");
}
}  // namespace wdc
