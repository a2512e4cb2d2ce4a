// Tensor-core split-sequence decode: the host-side plan (tensor maps, splits per CTA, heads per
// compute warp) and the head-dim-128 kernels of groups of up to 8 heads; the kernel itself is in
// kl_decode_tc_kernel.cuh, the head-dim-64 kernels in kl_decode_tc64.cu, those of larger groups
// in kl_decode_tc_groups.cu.
#include "kl_decode_tc_kernel.cuh"

namespace kl {
namespace {

template <bool kStandard, int KH, bool kExact>
cudaError_t launch_waits(const DecodeArgs &la, bool per_split, const CUtensorMap &vmap,
                         const CUtensorMap &kmap, const CUtensorMap &wmap, const CUtensorMap &qmap) {
    if (la.geo.D == 64)
        return launch_tc_head64(la, per_split, kStandard, KH, kExact, vmap, kmap, wmap, qmap);
    return launch_dim<kStandard, KH, kExact, false>(la, per_split, vmap, kmap, wmap, qmap);
}

template <bool kStandard>
cudaError_t launch(const DecodeArgs &a) {
    DecodeArgs la = a;
    const Geometry &g = la.geo;
    // cache viewed as [num_pages * Hkv * P rows][128]; one box = one page of one head
    const uint64_t cache_rows = (uint64_t)g.num_pages * g.Hkv * g.P;
    CUtensorMap vmap, kmap, wmap, qmap;
    if (!make_map(&vmap, a.v_cache, g.D, cache_rows, (uint32_t)g.P)) return cudaErrorInvalidValue;
    kmap = wmap = qmap = vmap;
    if (kStandard && !make_map(&kmap, a.k_cache, g.D, cache_rows, (uint32_t)g.P))
        return cudaErrorInvalidValue;
    if (!kStandard && !a.q_routed && a.w_r) {
        // W^R [Hw * 128 rows (k)][128 (j)], Hw = Hkv or Hq, one box = one 64-column half of one
        // matrix; q [B * Hq rows][128], one box = the up to 8 rows of one CTA's heads.
        const uint64_t hw = g.wr_per_qh ? (uint64_t)g.Hq : (uint64_t)g.Hkv;
        if (!make_map(&wmap, a.w_r, g.D, hw * g.D, (uint32_t)g.D)) return cudaErrorInvalidValue;
        if (!make_map(&qmap, a.q, g.D, (uint64_t)g.B * g.Hq, (uint32_t)g.qbox))
            return cudaErrorInvalidValue;
    }
    // Splits per CTA: one, unless one CTA per split would overflow a wave of two CTAs per SM
    // while the (b, g) units alone would not fill it (few long sequences split many ways): then
    // the fewest consecutive splits per CTA that fit the wave.
    const int64_t units = (int64_t)g.B * (g.Hkv / g.vpc) * g.nhb;
    const int64_t slots = 2 * (int64_t)device_sm_count();
    int spc = 1;
    if (g.S > 1 && units < slots)
        while ((int64_t)((g.S + spc - 1) / spc) * units > slots) ++spc;
    la.geo.spc = spc;
    const bool per_split = spc > 1 && !a.merge_inside && !a.direct_out;
    // heads per compute warp: all 8 (padded) on four warps; 4 on eight for the sibling CTAs
    // of larger groups (head dim 128); 2 on eight when the group has at most 4. Exact short
    // waits only when the limit asks for them.
    const bool exact = a.wait_ns < kExactWaitNs;
    if (g.nhb > 1 && g.D == 128)
        return launch_tc_groups(la, per_split, kStandard, exact, vmap, kmap, wmap, qmap);
    if (g.vpc * (g.G < kNG ? g.G : kNG) <= 4)
        return exact ? launch_waits<kStandard, 2, true>(la, per_split, vmap, kmap, wmap, qmap)
                     : launch_waits<kStandard, 2, false>(la, per_split, vmap, kmap, wmap, qmap);
    return exact ? launch_waits<kStandard, 8, true>(la, per_split, vmap, kmap, wmap, qmap)
                 : launch_waits<kStandard, 8, false>(la, per_split, vmap, kmap, wmap, qmap);
}

}  // namespace

bool tc_merge_inside(const Geometry &g, bool standard) {
    // the merging CTA keeps {m, l} and the weights of its heads' S states (12 B each) in its
    // ring and streams the state rows (512 B) through the rest, at least one split per round
    const size_t gc = g.vpc * g.G < kNG ? g.vpc * g.G : kNG;
    const size_t table = (gc * g.S * 12 + 1023) & ~(size_t)1023;
    const size_t ring = standard ? sizeof(Smem<true>::tiles) : sizeof(Smem<false>::tiles);
    return g.S > 1 && table + gc * kD * sizeof(float) <= ring;
}

bool tc_supported(const Geometry &g, bool standard) {
    (void)standard;
    if ((g.D != kD && g.D != 64) || g.G > kMaxGroup) return false;
    if (g.P != 16 && g.P != 32 && g.P != 64 && g.P != 128) return false;
    if ((int64_t)g.num_pages * g.Hkv * g.P >= ((int64_t)1 << 31)) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3;
}

cudaError_t launch_decode_tc(const DecodeArgs &a, bool standard) {
    if (a.geo.B == 0) return cudaSuccess;
    return standard ? launch<true>(a) : launch<false>(a);
}

}  // namespace kl
