// Host packer: pattern projection, connectivity pruning, filter grouping and the compact layout.
//
//  * projection onto the pattern set (§4.3, Eq. 6): per kernel, the pattern whose pruned kernel
//    keeps the largest Frobenius norm; scores in float64, ((a^2 + b^2) + c^2) + d^2 over the
//    pattern's taps in ascending raster order, ties to the lowest pattern index;
//  * connectivity pruning (§4.4, C'_n: at most beta nonzero kernels): the beta kernels with the
//    largest retained energy survive, ties to the lower flat index;
//  * filter kernel reorder and compressed weight storage (§3.4): filters sorted by
//    (kept count desc, pattern sequence asc, index asc) and dealt to groups of 8 in snake order
//    (balanced kept counts per group); per (group, ci) a 64-bit descriptor of (slot, pattern)
//    codes; 4 fp32 values per kept kernel.
//
// Built with -ffp-contract=off: every float64 operation below rounds on its own.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>

#include "../../include/patconv.h"
#include "layer.h"

using namespace patconv;

namespace {

int popcount9(unsigned m) {
    int c = 0;
    for (int t = 0; t < 9; ++t) c += (m >> t) & 1u;
    return c;
}

int taps_of(unsigned mask, int* taps) {
    int n = 0;
    for (int t = 0; t < 9; ++t)
        if ((mask >> t) & 1u) taps[n++] = t;
    return n;
}

int build(pp_layer* L, const float* W, double keep) {
    const int cout = L->cout, cin_g = L->cin_g, m = L->n_patterns;
    const size_t K = (size_t)cout * (size_t)cin_g;

    int taps[kMaxPatterns][4];
    for (int p = 0; p < m; ++p) taps_of(L->masks[p], taps[p]);

    // 1. projection: best pattern and its retained energy per kernel
    std::vector<int> best(K);
    std::vector<double> retained(K);
    for (size_t k = 0; k < K; ++k) {
        const float* w = W + 9 * k;
        int bp = 0;
        double bs = -1.0;
        for (int p = 0; p < m; ++p) {
            double s = 0.0;
            for (int j = 0; j < 4; ++j) {
                const double v = (double)w[taps[p][j]];
                const double sq = v * v;
                s = (j == 0) ? sq : s + sq;
            }
            if (s > bs) { bs = s; bp = p; }
        }
        best[k] = bp;
        retained[k] = bs;
    }

    // 2. connectivity: beta = floor(keep*K + 0.5), clamp [1, K]; rank (energy desc, index asc)
    const double prod = keep * (double)K;
    const double rounded = std::floor(prod + 0.5);
    long long beta = (long long)rounded;
    if (beta < 1) beta = 1;
    if (beta > (long long)K) beta = (long long)K;
    L->beta = (int)beta;

    std::vector<uint32_t> order(K);
    for (size_t k = 0; k < K; ++k) order[k] = (uint32_t)k;
    std::sort(order.begin(), order.end(), [&](uint32_t a, uint32_t b) {
        if (retained[a] != retained[b]) return retained[a] > retained[b];
        return a < b;
    });
    L->pid.assign(K, (int8_t)-1);
    for (long long i = 0; i < beta; ++i) L->pid[order[i]] = (int8_t)best[order[i]];

    // 3. filter kernel reorder: (kept count desc, pattern sequence asc (pruned = 15), index asc)
    std::vector<int> count(cout, 0);
    for (int co = 0; co < cout; ++co)
        for (int ci = 0; ci < cin_g; ++ci) count[co] += L->pid[(size_t)co * cin_g + ci] >= 0;
    std::vector<int> fo(cout);
    for (int co = 0; co < cout; ++co) fo[co] = co;
    auto seq = [&](int co, int ci) {
        const int p = L->pid[(size_t)co * cin_g + ci];
        return p < 0 ? 15 : p;
    };
    std::sort(fo.begin(), fo.end(), [&](int a, int b) {
        if (count[a] != count[b]) return count[a] > count[b];
        for (int ci = 0; ci < cin_g; ++ci) {
            const int sa = seq(a, ci), sb = seq(b, ci);
            if (sa != sb) return sa < sb;
        }
        return a < b;
    });

    // deal the sorted filters over the G groups in snake order (round r fills slot r of every
    // group, alternating direction), so that every group gets a similar number of kept kernels:
    // one warp processes one group, and the warps of a CTA then finish their channels together
    const int G = (cout + kF - 1) / kF;
    L->G = G;
    L->perm.assign((size_t)G * kF, kPadSlot);
    for (int j = 0; j < cout; ++j) {
        const int round = j / G, pos = j % G;
        const int g = (round % 2 == 0) ? pos : G - 1 - pos;
        L->perm[(size_t)g * kF + round] = (uint32_t)fo[j];
    }

    // 4. compressed weight storage
    L->desc.assign((size_t)G * cin_g, 0);
    L->kofs.assign((size_t)G * cin_g + 1, 0);
    L->vals.clear();
    L->vals.reserve((size_t)beta * 4);
    uint32_t n = 0;
    for (int g = 0; g < G; ++g) {
        for (int ci = 0; ci < cin_g; ++ci) {
            L->kofs[(size_t)g * cin_g + ci] = n;
            uint64_t word = 0;
            unsigned c = 0;
            for (int f = 0; f < kF; ++f) {
                const uint32_t co_u = L->perm[(size_t)g * kF + f];
                if (co_u == kPadSlot) continue;
                const int co = (int)co_u;
                const int p = L->pid[(size_t)co * cin_g + ci];
                if (p < 0) continue;
                word |= (uint64_t)((unsigned)(f << 3) | (unsigned)p) << (4 + 6 * c);
                ++c;
                const float* w = W + 9 * ((size_t)co * cin_g + ci);
                for (int t = 0; t < 4; ++t) L->vals.push_back(w[taps[p][t]]);
                ++n;
            }
            L->desc[(size_t)g * cin_g + ci] = word | c;
        }
    }
    L->kofs[(size_t)G * cin_g] = n;

    // 5. header, dense projected weights, device image
    L->header.assign(16, 0);
    const uint32_t hv[10] = {kMagic, kVersion, (uint32_t)cout, (uint32_t)cin_g,
                             (uint32_t)L->groups, (uint32_t)L->stride, (uint32_t)m,
                             (uint32_t)beta, (uint32_t)kF, (uint32_t)G};
    for (int i = 0; i < 10; ++i) L->header[i] = hv[i];
    for (int i = 0; i < 4; ++i)
        L->header[10 + i] = (uint32_t)L->masks[2 * i] | ((uint32_t)L->masks[2 * i + 1] << 16);

    L->dense.assign(K * 9, 0.0f);
    for (size_t k = 0; k < K; ++k) {
        const int p = L->pid[k];
        if (p < 0) continue;
        for (int j = 0; j < 4; ++j) L->dense[9 * k + taps[p][j]] = W[9 * k + taps[p][j]];
    }

    const size_t b_perm = L->perm.size() * 4, b_desc = L->desc.size() * 8,
                 b_kofs = L->kofs.size() * 4, b_vals = L->vals.size() * 4;
    L->off_perm = 0;
    L->off_desc = align256(b_perm);
    L->off_kofs = L->off_desc + align256(b_desc);
    L->off_vals = L->off_kofs + align256(b_kofs);
    L->image.assign(L->off_vals + align256(b_vals), 0);
    std::memcpy(L->image.data() + L->off_perm, L->perm.data(), b_perm);
    std::memcpy(L->image.data() + L->off_desc, L->desc.data(), b_desc);
    std::memcpy(L->image.data() + L->off_kofs, L->kofs.data(), b_kofs);
    if (b_vals) std::memcpy(L->image.data() + L->off_vals, L->vals.data(), b_vals);
    return PP_OK;
}

size_t section_bytes(const pp_layer* L, int s) {
    switch (s) {
        case PP_SEC_HEADER: return L->header.size() * 4;
        case PP_SEC_PID: return L->pid.size();
        case PP_SEC_PERM: return L->perm.size() * 4;
        case PP_SEC_DESC: return L->desc.size() * 8;
        case PP_SEC_KOFS: return L->kofs.size() * 4;
        case PP_SEC_VALS: return L->vals.size() * 4;
        case PP_SEC_DENSE: return L->dense.size() * 4;
        case PP_SEC_IMAGE: return L->image.size();
        default: return (size_t)-1;
    }
}

const void* section_data(const pp_layer* L, int s) {
    switch (s) {
        case PP_SEC_HEADER: return L->header.data();
        case PP_SEC_PID: return L->pid.data();
        case PP_SEC_PERM: return L->perm.data();
        case PP_SEC_DESC: return L->desc.data();
        case PP_SEC_KOFS: return L->kofs.data();
        case PP_SEC_VALS: return L->vals.data();
        case PP_SEC_DENSE: return L->dense.data();
        case PP_SEC_IMAGE: return L->image.data();
        default: return nullptr;
    }
}

}  // namespace

extern "C" {

int pp_default_patterns(uint16_t* masks, int capacity) {
    if (capacity > 0 && !masks) return PP_ERR_NULL;
    for (int i = 0; i < capacity && i < kMaxPatterns; ++i) masks[i] = kDefaultMasks[i];
    return kMaxPatterns;
}

int pp_design_patterns(const float* W, size_t n_kernels, int m, uint16_t* masks, int* n_masks) {
    if (!W || !masks || !n_masks) return PP_ERR_NULL;
    if (n_kernels == 0 || m < 1 || m > kMaxPatterns) return PP_ERR_SHAPE;
    // candidate pattern of every kernel: the centre and the three non-central taps of largest
    // magnitude (equal magnitudes: the lower tap first); a mask is a 9-bit integer < 512
    std::vector<uint64_t> count(512, 0);
    for (size_t k = 0; k < n_kernels; ++k) {
        const float* w = W + 9 * k;
        for (int t = 0; t < 9; ++t)
            if (!std::isfinite(w[t])) return PP_ERR_NONFINITE;
        uint32_t mask = 1u << 4;
        for (int pick = 0; pick < 3; ++pick) {
            int best = -1;
            for (int t = 0; t < 9; ++t) {
                if (mask >> t & 1u) continue;
                if (best < 0 || std::fabs(w[t]) > std::fabs(w[best])) best = t;
            }
            mask |= 1u << best;
        }
        ++count[mask];
    }
    // the m most frequent candidates, by count descending, then by mask value ascending
    std::vector<int> order;
    for (int mk = 0; mk < 512; ++mk)
        if (count[mk]) order.push_back(mk);
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return count[a] > count[b]; });
    const int n = std::min<int>(m, (int)order.size());
    for (int i = 0; i < n; ++i) masks[i] = (uint16_t)order[i];
    *n_masks = n;
    return PP_OK;
}

int pp_pack(const float* W, int Cout, int Cin, int groups, int stride, const uint16_t* masks,
            int n_patterns, double keep, pp_handle* out) {
    if (!W || !masks || !out) return PP_ERR_NULL;
    if (Cout < 1 || Cin < 1) return PP_ERR_SHAPE;
    if (!(groups == 1 || (groups == Cin && groups == Cout))) return PP_ERR_SHAPE;
    if (stride != 1 && stride != 2) return PP_ERR_SHAPE;
    const int cin_g = groups == 1 ? Cin : 1;
    if ((long long)Cout * cin_g > (1LL << 30)) return PP_ERR_SHAPE;
    if (n_patterns < 1 || n_patterns > kMaxPatterns) return PP_ERR_PATTERN;
    for (int i = 0; i < n_patterns; ++i) {
        if (masks[i] >= 512 || popcount9(masks[i]) != 4) return PP_ERR_PATTERN;
        for (int j = 0; j < i; ++j)
            if (masks[i] == masks[j]) return PP_ERR_PATTERN;
    }
    if (!(keep > 0.0 && keep <= 1.0)) return PP_ERR_KEEP;
    const size_t nw = (size_t)Cout * cin_g * 9;
    for (size_t i = 0; i < nw; ++i)
        if (!std::isfinite(W[i])) return PP_ERR_NONFINITE;

    pp_layer* L = new (std::nothrow) pp_layer();
    if (!L) return PP_ERR_ALLOC;
    L->cout = Cout;
    L->cin_g = cin_g;
    L->groups = groups;
    L->depthwise = groups != 1;
    L->stride = stride;
    L->n_patterns = n_patterns;
    bool fast = n_patterns == kMaxPatterns;
    for (int i = 0; i < n_patterns; ++i) {
        L->masks[i] = masks[i];
        fast = fast && masks[i] == kDefaultMasks[i];
    }
    L->fast = fast;
    int st;
    try {
        st = build(L, W, keep);
    } catch (const std::bad_alloc&) {
        st = PP_ERR_ALLOC;
    }
    if (st != PP_OK) {
        delete L;
        return st;
    }
    *out = L;
    return PP_OK;
}

int pp_query(pp_handle h, int key, int64_t* value) {
    if (!h || !value) return PP_ERR_NULL;
    int64_t v;
    switch (key) {
        case PP_Q_BETA: v = h->beta; break;
        case PP_Q_COUT: v = h->cout; break;
        case PP_Q_CIN_G: v = h->cin_g; break;
        case PP_Q_GROUPS: v = h->groups; break;
        case PP_Q_STRIDE: v = h->stride; break;
        case PP_Q_N_GROUPS: v = h->G; break;
        case PP_Q_N_PATTERNS: v = h->n_patterns; break;
        case PP_Q_IMAGE_BYTES: v = (int64_t)h->image.size(); break;
        case PP_Q_FAST_PATH: v = h->fast ? 1 : 0; break;
        default:
            if (key >= PP_Q_SECTION_BYTES && key <= PP_Q_SECTION_BYTES + PP_SEC_IMAGE) {
                v = (int64_t)section_bytes(h, key - PP_Q_SECTION_BYTES);
                break;
            }
            return PP_ERR_ARG;
    }
    *value = v;
    return PP_OK;
}

int pp_export(pp_handle h, int section, void* host_dst, size_t bytes) {
    if (!h) return PP_ERR_NULL;
    if (section < PP_SEC_HEADER || section > PP_SEC_IMAGE) return PP_ERR_ARG;
    const size_t n = section_bytes(h, section);
    if (bytes != n) return PP_ERR_BUFFER;
    if (n == 0) return PP_OK;
    if (!host_dst) return PP_ERR_NULL;
    std::memcpy(host_dst, section_data(h, section), n);
    return PP_OK;
}

int pp_destroy(pp_handle h) {
    delete h;
    return PP_OK;
}

const char* pp_status_string(int status) {
    switch (status) {
        case PP_OK: return "ok";
        case PP_ERR_NULL: return "null pointer argument";
        case PP_ERR_SHAPE: return "size out of range or inconsistent";
        case PP_ERR_PATTERN: return "invalid pattern library (1..8 distinct 4-tap 9-bit masks)";
        case PP_ERR_KEEP: return "keep ratio outside (0, 1]";
        case PP_ERR_NONFINITE: return "non-finite weight";
        case PP_ERR_ALIGN: return "device pointer misaligned";
        case PP_ERR_DTYPE: return "unknown dtype";
        case PP_ERR_NOT_BOUND: return "layer not bound to a device image";
        case PP_ERR_BUFFER: return "buffer size mismatch or overlapping buffers";
        case PP_ERR_CUDA: return "CUDA runtime error";
        case PP_ERR_ARG: return "invalid argument";
        case PP_ERR_ALLOC: return "host allocation failed";
        case PP_ERR_SCRATCH: return "call needs more scratch than the library's static scratch array holds";
        case PP_ERR_PATH: return "the layer's kernel does not offer this fusion (dense layers of the compiled pattern library only)";
        default: return "unknown status";
    }
}

}  // extern "C"
