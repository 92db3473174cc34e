// Tensor-map encoding with a cache: a layer call needs about two dozen maps
// whose encoding is pure host work, repeated identically from call to call.
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>
#include <unordered_map>

#include "tmap.h"

namespace mosa {
namespace {

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

struct Key {
    uint64_t dtype;
    uint64_t base;
    uint64_t dims[5], strides[4];
    uint32_t box[5];
    int rank;
    bool operator==(const Key &o) const { return std::memcmp(this, &o, sizeof(Key)) == 0; }
};

struct KeyHash {
    size_t operator()(const Key &k) const {
        const uint64_t *w = reinterpret_cast<const uint64_t *>(&k);
        uint64_t h = 1469598103934665603ull;
        for (size_t i = 0; i < sizeof(Key) / 8; ++i) h = (h ^ w[i]) * 1099511628211ull;
        return (size_t)h;
    }
};

std::mutex g_mu;
std::unordered_map<Key, CUtensorMap, KeyHash> g_cache;
constexpr size_t kMaxEntries = 4096;

}  // namespace

bool tmap_available() { return encoder() != nullptr; }

namespace {

bool encode(CUtensorMapDataType dtype, CUtensorMap *out, const void *base, int rank,
            const uint64_t *dims, const uint64_t *strides, const uint32_t *box) {
    if (rank < 1 || rank > 5) return false;
    Key key;
    std::memset(&key, 0, sizeof(key));
    key.dtype = (uint64_t)dtype;
    key.base = reinterpret_cast<uint64_t>(base);
    key.rank = rank;
    for (int i = 0; i < rank; ++i) {
        key.dims[i] = dims[i];
        key.box[i] = box[i];
    }
    for (int i = 0; i < rank - 1; ++i) key.strides[i] = strides[i];
    {
        std::lock_guard<std::mutex> lk(g_mu);
        auto it = g_cache.find(key);
        if (it != g_cache.end()) {
            *out = it->second;
            return true;
        }
    }
    auto fn = encoder();
    if (!fn) return false;
    cuuint64_t gd[5], gs[4];
    cuuint32_t bx[5], es[5] = {1, 1, 1, 1, 1};
    for (int i = 0; i < rank; ++i) {
        gd[i] = dims[i];
        bx[i] = box[i];
    }
    for (int i = 0; i < rank - 1; ++i) gs[i] = strides[i];
    CUtensorMap m;
    if (fn(&m, dtype, (cuuint32_t)rank, const_cast<void *>(base), gd,
           gs, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return false;
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_cache.size() >= kMaxEntries) g_cache.clear();
    g_cache.emplace(key, m);
    *out = m;
    return true;
}

}  // namespace

bool tmap_bf16(CUtensorMap *out, const void *base, int rank, const uint64_t *dims,
               const uint64_t *strides, const uint32_t *box) {
    return encode(CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, out, base, rank, dims, strides, box);
}

bool tmap_f32(CUtensorMap *out, const void *base, int rank, const uint64_t *dims,
              const uint64_t *strides, const uint32_t *box) {
    return encode(CU_TENSOR_MAP_DATA_TYPE_FLOAT32, out, base, rank, dims, strides, box);
}

}  // namespace mosa
