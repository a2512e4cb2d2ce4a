// Head-dim-64 instances of the tensor-core decode (the kernel is in kl_decode_tc_kernel.cuh):
// compiled in their own translation unit, in parallel with the head-dim-128 ones.
#include "kl_decode_tc_kernel.cuh"

namespace kl {

cudaError_t launch_tc_head64(const DecodeArgs &la, bool per_split, bool standard, int KH, bool exact,
                             const CUtensorMap &vmap, const CUtensorMap &kmap,
                             const CUtensorMap &wmap, const CUtensorMap &qmap) {
    if (standard) {
        if (KH == 2)
            return exact ? launch_dim<true, 2, true, true>(la, per_split, vmap, kmap, wmap, qmap)
                         : launch_dim<true, 2, false, true>(la, per_split, vmap, kmap, wmap, qmap);
        return exact ? launch_dim<true, 8, true, true>(la, per_split, vmap, kmap, wmap, qmap)
                     : launch_dim<true, 8, false, true>(la, per_split, vmap, kmap, wmap, qmap);
    }
    if (KH == 2)
        return exact ? launch_dim<false, 2, true, true>(la, per_split, vmap, kmap, wmap, qmap)
                     : launch_dim<false, 2, false, true>(la, per_split, vmap, kmap, wmap, qmap);
    return exact ? launch_dim<false, 8, true, true>(la, per_split, vmap, kmap, wmap, qmap)
                 : launch_dim<false, 8, false, true>(la, per_split, vmap, kmap, wmap, qmap);
}

}  // namespace kl
