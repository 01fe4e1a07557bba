// Host-side state of one packed layer, shared by the packer (pack.cpp) and the CUDA launchers
// (conv.cu).  Not part of the public ABI (include/patconv.h).
#pragma once

#include <cstddef>
#include <cstdint>
#include <memory>
#include <mutex>
#include <vector>

namespace patconv {

constexpr int kF = 8;                 // filters per group (slots per warp)
constexpr int kMaxPatterns = 8;
constexpr uint32_t kPadSlot = 0xFFFFFFFFu;
constexpr uint32_t kMagic = 0x314B5050u;  // 'PPK1'
constexpr uint32_t kVersion = 1;

// The compiled pattern library, raster taps (bit t = tap 3*(dy+1)+(dx+1)):
//   0 {3,4,5,7}  1 {1,4,5,7}  2 {1,3,4,7}  3 {1,3,4,5}   centre + 3 of the 4 edge neighbours
//   4 {0,1,2,4}  5 {0,3,4,6}  6 {2,4,5,8}  7 {4,6,7,8}   centre + edge + its 2 flanking corners
constexpr uint16_t kDefaultMasks[kMaxPatterns] = {0x0B8, 0x0B2, 0x09A, 0x03A,
                                                  0x017, 0x059, 0x134, 0x1D0};

inline size_t align256(size_t n) { return (n + 255) / 256 * 256; }

// Launch plans the CUDA side caches per handle (defined in conv.cu; destroyed with the handle).
struct PlanCacheBase {
    virtual ~PlanCacheBase() = default;
};

}  // namespace patconv

struct pp_layer {
    int cout = 0, cin_g = 0, groups = 1, stride = 1, n_patterns = 0, beta = 0, G = 0;
    uint16_t masks[patconv::kMaxPatterns] = {};
    bool fast = false;                 // masks == kDefaultMasks (compiled pattern bodies)
    bool depthwise = false;

    std::vector<uint32_t> header;      // u32[16]
    std::vector<int8_t> pid;           // [cout][cin_g], -1 = pruned
    std::vector<uint32_t> perm;        // [G*8]
    std::vector<uint64_t> desc;        // [G*cin_g]
    std::vector<uint32_t> kofs;        // [G*cin_g + 1]
    std::vector<float> vals;           // [beta*4]
    std::vector<float> dense;          // [cout*cin_g*9]
    std::vector<uint8_t> image;        // perm | desc | kofs | vals, 256-B aligned sections
    size_t off_perm = 0, off_desc = 0, off_kofs = 0, off_vals = 0;

    void* dev = nullptr;               // caller-owned device copy of `image`
    size_t dev_bytes = 0;

    // launch plans by call shape (conv.cu), created on the first plan by call_once, so that calls
    // from several host threads see it fully constructed
    std::unique_ptr<patconv::PlanCacheBase> plans;
    std::once_flag plans_once;
};
