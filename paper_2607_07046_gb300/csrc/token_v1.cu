// Decode-token kernel variants for the 7B (D 4096, MHA), 8B (D 4096, 4 query heads per KV head)
// and 13B (D 5120, shards with different O row lengths) shapes.
#include "token_kernel.cuh"

namespace vt {

int token_variants_workloads(const TokVariant** out) {
    static const TokVariant v[] = {
        TokVariantImpl<8, 2, 128, 1, false>::desc(),
        TokVariantImpl<8, 2, 128, 4, false>::desc(),
        TokVariantImpl<10, 3, 128, 1, true>::desc(),
    };
    *out = v;
    return (int)(sizeof(v) / sizeof(v[0]));
}

}  // namespace vt
