// tcgen05 flash attention (placeholder until the TMEM kernel lands).
#include "dit_kernels.cuh"
namespace wdc {
bool tc_attention_supported(int, int) { return false; }
wdc_status tc_attention(Ctx* c, const void*, const void*, const void*, void*, int, int, int, cudaStream_t) {
    return fail(c, WDC_ERR_UNSUPPORTED, "tcgen05 attention not built");
}
}  // namespace wdc
