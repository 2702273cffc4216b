// Decode-token kernel variants for small models (D 256 to 1024, head dim 64 or 128).
#include "token_kernel.cuh"

namespace vt {

int token_variants_small(const TokVariant** out) {
    static const TokVariant v[] = {
        TokVariantImpl<4, 1, 64, 1, true>::desc(),  TokVariantImpl<4, 1, 64, 2, true>::desc(),
        TokVariantImpl<2, 1, 64, 2, true>::desc(),  TokVariantImpl<8, 1, 128, 1, true>::desc(),
        TokVariantImpl<8, 1, 128, 4, true>::desc(),
    };
    *out = v;
    return (int)(sizeof(v) / sizeof(v[0]));
}

}  // namespace vt
