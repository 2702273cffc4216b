// Prefill-path kernels (dense prompt): placeholder until the tensor-core path lands.
#include "internal.h"

namespace vt {

cudaError_t init_prefill_kernels() { return cudaSuccess; }

vt_status prefill_attn_shard(const PrefillAttnArgs&, cudaStream_t, std::string* err) {
    *err = "prefill is not available in this build";
    return VT_ERR_STATE;
}

vt_status prefill_ffn_shard(const PrefillFfnArgs&, cudaStream_t, std::string* err) {
    *err = "prefill is not available in this build";
    return VT_ERR_STATE;
}

}  // namespace vt
