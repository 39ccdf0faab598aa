// Decode-step attention over the kept cache with mixed-precision values: the reserved values (R_V and the
// recency buffer) in bf16, every other kept value read back from its b-bit codes (the quantizer of Sec. 4.4,
// the reserved cache proposed in Sec. 6).  The CUDA-core kernel of decode_simt.cuh with kBits = 2, 4 or 8:
// each chunk brings K rows, code rows and (s, z) by bulk copies, the bf16 rows of its reserved slots by one bulk
// copy from the reserved cache (where they follow each other in slot order), and the rows of slots appended
// since the quantization by one more.
#include <algorithm>
#include <cfloat>
#include <map>
#include <mutex>
#include <tuple>

#include "kernels.cuh"
#include "ptx.cuh"

namespace vase {

namespace {

#include "decode_simt.cuh"

template <int Gp, int kBits>
cudaError_t launch_kernel(const DecodeParams& p, size_t smem, cudaStream_t s) {
    return simt::launch_gp<Gp, kBits>(p, smem, s);
}

template <int Gp, int kBits>
const void* kernel_fn() {
    return reinterpret_cast<const void*>(simt::decode_simt_kernel<Gp, kBits>);
}

template <int Gp>
cudaError_t set_attributes_gp() {
    cudaError_t e = cudaSuccess;
    const int a2 = static_cast<int>(simt::decode_layout(Gp, 2, kDecodeMaxMaskWords).total);
    const int a4 = static_cast<int>(simt::decode_layout(Gp, 4, kDecodeMaxMaskWords).total);
    const int a8 = static_cast<int>(simt::decode_layout(Gp, 8, kDecodeMaxMaskWords).total);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(simt::decode_simt_kernel<Gp, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, a2);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(simt::decode_simt_kernel<Gp, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, a4);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(simt::decode_simt_kernel<Gp, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, a8);
    return e;
}

int padded_gp(int G) { return G <= 2 ? 2 : G <= 4 ? 4 : 8; }

}  // namespace

size_t decode_mixed_smem_bytes(int G, int bits, int mask_words) {
    return simt::decode_layout(padded_gp(G), bits, mask_words).total;
}

cudaError_t decode_mixed_set_attributes() {
    cudaError_t e = set_attributes_gp<2>();
    if (e == cudaSuccess) e = set_attributes_gp<4>();
    if (e == cudaSuccess) e = set_attributes_gp<8>();
    return e;
}

namespace {

const void* mixed_kernel(int Gp, int bits) {
    if (Gp == 2) return bits == 2 ? kernel_fn<2, 2>() : bits == 4 ? kernel_fn<2, 4>() : kernel_fn<2, 8>();
    if (Gp == 4) return bits == 2 ? kernel_fn<4, 2>() : bits == 4 ? kernel_fn<4, 4>() : kernel_fn<4, 8>();
    return bits == 2 ? kernel_fn<8, 2>() : bits == 4 ? kernel_fn<8, 4>() : kernel_fn<8, 8>();
}

// CTAs per unit: the largest cluster size (at most kDecodeMaxCluster and the unit's chunks) whose clusters all
// fit on the GPU at once, asked of the occupancy calculator (clusters must fit within one GPC, so the count
// depends on the GPCs' sizes, not only on the SM count).  Results are kept per launch shape.
int mixed_cluster(int Gp, int bits, size_t smem, int units, int n_chunks) {
    static std::mutex mu;
    static std::map<std::tuple<int, int, size_t, int, int>, int> memo;
    const auto key = std::make_tuple(Gp, bits, smem, units, n_chunks);
    std::lock_guard<std::mutex> lock(mu);
    auto it = memo.find(key);
    if (it != memo.end()) return it->second;
    int best = 1;
    for (int c = std::min(kDecodeMaxCluster, n_chunks); c >= 1; --c) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(c), static_cast<unsigned>(units));
        cfg.blockDim = dim3(simt::kThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = static_cast<unsigned>(c);
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int active = 0;
        if (cudaOccupancyMaxActiveClusters(&active, mixed_kernel(Gp, bits), &cfg) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        if (active >= units) {
            best = c;
            break;
        }
    }
    memo[key] = best;
    return best;
}

}  // namespace

// Returns cudaErrorInvalidValue when the unit's masks exceed kDecodeMaxMaskWords (more than 17408 slots) or G > 8.
cudaError_t launch_decode_mixed(DecodeParams p, int num_sms, cudaStream_t s) {
    (void)num_sms;
    if (p.G > 8 || p.mask_words > kDecodeMaxMaskWords) return cudaErrorInvalidValue;
    const int Gp = padded_gp(p.G);
    const size_t smem = decode_mixed_smem_bytes(p.G, p.bits, p.mask_words);
    p.n_chunks = (p.fill + simt::kChunk - 1) / simt::kChunk;
    p.cluster = mixed_cluster(Gp, p.bits, smem, p.units, p.n_chunks);
    if (Gp == 2) return p.bits == 2 ? launch_kernel<2, 2>(p, smem, s) : p.bits == 4 ? launch_kernel<2, 4>(p, smem, s)
                                                                                  : launch_kernel<2, 8>(p, smem, s);
    if (Gp == 4) return p.bits == 2 ? launch_kernel<4, 2>(p, smem, s) : p.bits == 4 ? launch_kernel<4, 4>(p, smem, s)
                                                                                  : launch_kernel<4, 8>(p, smem, s);
    return p.bits == 2 ? launch_kernel<8, 2>(p, smem, s) : p.bits == 4 ? launch_kernel<8, 4>(p, smem, s)
                                                                     : launch_kernel<8, 8>(p, smem, s);
}

}  // namespace vase
