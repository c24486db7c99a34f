// attn_fp8.cu -- node-chunk attention for e4m3 KV (written after the bf16 path).
#include "internal.h"

namespace parason {

cudaError_t launch_attn_fp8(const AttnArgs &, const CUtensorMap &, const CUtensorMap &, int,
                            cudaStream_t) {
    return cudaErrorNotSupported;
}

}  // namespace parason
