// Head-dim-128 instances of the tensor-core decode for the sibling CTAs of groups of more than
// 8 query heads (4 heads on each of eight compute warps; the kernel is in
// kl_decode_tc_kernel.cuh): compiled in their own translation unit, in parallel with the others.
#include "kl_decode_tc_kernel.cuh"

namespace kl {

cudaError_t launch_tc_groups(const DecodeArgs &la, bool per_split, bool standard, bool exact,
                             const CUtensorMap &vmap, const CUtensorMap &kmap,
                             const CUtensorMap &wmap, const CUtensorMap &qmap) {
    if (standard)
        return exact ? launch_dim<true, 4, true, false>(la, per_split, vmap, kmap, wmap, qmap)
                     : launch_dim<true, 4, false, false>(la, per_split, vmap, kmap, wmap, qmap);
    return exact ? launch_dim<false, 4, true, false>(la, per_split, vmap, kmap, wmap, qmap)
                 : launch_dim<false, 4, false, false>(la, per_split, vmap, kmap, wmap, qmap);
}

}  // namespace kl
