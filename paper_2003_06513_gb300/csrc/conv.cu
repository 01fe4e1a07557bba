// CUDA kernels and launchers of libpatconv (sm_103a): pattern-sparse 3x3 convolution.
//
// Work decomposition of the main kernel (pconv_main):
//   * a lane owns an RY x RX block of output pixels of one image;
//   * a warp owns one filter group (8 filters, "filter kernel reorder" of §3.4) for the 32
//     blocks of its CTA's spatial tile and keeps 8 x RY*RX fp32 accumulators in registers;
//   * a CTA is 8 warps = 8 filter groups (64 filters) over one spatial tile, so every input
//     element staged in shared memory is reused by 64 filters;
//   * input channels stream through a multi-stage cp.async pipeline: the tile of CK channels,
//     with its zero halo (padding 1), lands in shared memory together with each group's
//     descriptors and kept weights for those channels;
//   * per input channel a lane loads its (RY-1)*S+3 x (RX-1)*S+3 input window into registers
//     once and applies it to every kept kernel of its group: the 6-bit (slot, pattern) code of
//     each kept kernel selects one of 64 compile-time bodies whose four tap offsets are
//     constants (the 4 taps of §3.2), so no per-element index is decoded;
//   * epilogue: + bias, ReLU, fp32 or fp16 (round to nearest even) vector stores to the
//     original channel of each slot.
// The path is a gathered sparse contraction, so it runs on the CUDA-core FFMA pipe.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <climits>
#include <cstdint>

#include "../../include/patconv.h"
#include "layer.h"

using namespace patconv;

namespace {

// ------------------------------------------------------------------------------ constants

// k-th tap (ascending raster order) of pattern p of the compiled library (kDefaultMasks).
__host__ __device__ constexpr int ktap(int p, int k) {
    const unsigned m = p == 0 ? 0x0B8u : p == 1 ? 0x0B2u : p == 2 ? 0x09Au : p == 3 ? 0x03Au
                     : p == 4 ? 0x017u : p == 5 ? 0x059u : p == 6 ? 0x134u : 0x1D0u;
    int n = 0;
    for (int t = 0; t < 9; ++t) {
        if ((m >> t) & 1u) {
            if (n == k) return t;
            ++n;
        }
    }
    return -1;
}

constexpr int kThreads = 256;   // 8 warps = 8 filter groups per CTA
constexpr int kWarps = kThreads / 32;
constexpr int kMaxBoundaries = 80;  // chunk boundaries cached per warp (C <= 79*CK)

struct MainParams {
    const void* x;
    void* y;
    const float* bias;
    const uint32_t* perm;
    const uint64_t* desc;
    const uint32_t* kofs;
    const float4* vals;
    int N, C, H, W, Cout, Ho, Wo, G, relu;
    int BY, BX, NB;                   // spatial tile: BY x BX blocks of NB images
    int tiles_x, tiles_y, tiles_n, n_fchunks;
    int CK, n_chunks;                 // input channels per pipeline stage, number of stages run
    int IH, IW, pitch;                // staged rows / cols per (channel, image), row pitch
    int vec_store;                    // y rows allow RX-wide vector stores
    int stage_floats;                 // input floats per stage
};

// ------------------------------------------------------------------------------ helpers

__device__ __forceinline__ void cp_async4(void* smem, const void* gmem, bool valid) {
    const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    const int n = valid ? 4 : 0;
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
    const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(s), "l"(gmem));
}
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem));
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__half>(__half v) { return __half2float(v); }

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __half from_f32<__half>(float v) { return __float2half_rn(v); }

// ------------------------------------------------------------------------------ main kernel

template <int S, int RY, int RX>
struct Win {
    static constexpr int WY = (RY - 1) * S + 3;
    static constexpr int WX = (RX - 1) * S + 3;
};

// acc[F_][*] += the pattern-P_ kernel (weights w) applied to the lane's input window.
template <int F_, int P_, int S, int RY, int RX, int WY, int WX>
__device__ __forceinline__ void fma_pattern(float (&acc)[kF][RY * RX], const float (&win)[WY][WX],
                                            const float4& w) {
    constexpr int t0 = ktap(P_, 0), t1 = ktap(P_, 1), t2 = ktap(P_, 2), t3 = ktap(P_, 3);
#pragma unroll
    for (int r = 0; r < RY; ++r) {
#pragma unroll
        for (int c = 0; c < RX; ++c) {
            float a = acc[F_][r * RX + c];
            a = fmaf(w.x, win[r * S + t0 / 3][c * S + t0 % 3], a);
            a = fmaf(w.y, win[r * S + t1 / 3][c * S + t1 % 3], a);
            a = fmaf(w.z, win[r * S + t2 / 3][c * S + t2 % 3], a);
            a = fmaf(w.w, win[r * S + t3 / 3][c * S + t3 % 3], a);
            acc[F_][r * RX + c] = a;
        }
    }
}

#define PP_CASE(F_, P_)                                                        \
    case ((F_) << 3) | (P_):                                                   \
        fma_pattern<F_, P_, S, RY, RX, WY, WX>(acc, win, w);                   \
        break;
#define PP_CASES(F_) \
    PP_CASE(F_, 0) PP_CASE(F_, 1) PP_CASE(F_, 2) PP_CASE(F_, 3) PP_CASE(F_, 4) PP_CASE(F_, 5) PP_CASE(F_, 6) PP_CASE(F_, 7)

template <int S, int RY, int RX, int WY, int WX>
__device__ __forceinline__ void dispatch(int code, const float4& w, float (&acc)[kF][RY * RX],
                                         const float (&win)[WY][WX]) {
    switch (code) {
        PP_CASES(0) PP_CASES(1) PP_CASES(2) PP_CASES(3)
        PP_CASES(4) PP_CASES(5) PP_CASES(6) PP_CASES(7)
        default: break;
    }
}

// Stage chunk `k` (channels [k*CK, k*CK+CK) ∩ [0, C)) into stage buffer `buf`.
template <typename TIn>
__device__ __forceinline__ void stage_chunk(const MainParams& p, int k, float* s_in, uint64_t* s_desc,
                                            float4* s_vals, const uint32_t* s_kb, int g, int n0,
                                            int iy0, int ix0) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c0 = k * p.CK;
    const int ckv = min(p.CK, p.C - c0);
    // input tile: rows of (cl, img, row) distributed over warps, columns over lanes
    const int rows = ckv * p.NB * p.IH;
    const TIn* x = static_cast<const TIn*>(p.x);
    for (int r = warp; r < rows; r += kWarps) {
        const int row = r % p.IH;
        const int t = r / p.IH;
        const int img = t % p.NB;
        const int cl = t / p.NB;
        const int n = n0 + img, ci = c0 + cl, iy = iy0 + row;
        const bool row_ok = n < p.N && iy >= 0 && iy < p.H;
        const size_t gbase = (((size_t)n * p.C + ci) * p.H + (row_ok ? iy : 0)) * p.W;
        float* srow = s_in + ((size_t)(cl * p.NB + img) * p.IH + row) * p.pitch;
        for (int c = lane; c < p.IW; c += 32) {
            const int ix = ix0 + c;
            const bool ok = row_ok && ix >= 0 && ix < p.W;
            if constexpr (sizeof(TIn) == 4) {
                cp_async4(srow + c, ok ? (const void*)(x + gbase + ix) : p.x, ok);
            } else {
                srow[c] = ok ? to_f32<TIn>(x[gbase + ix]) : 0.0f;
            }
        }
    }
    // this warp's group: descriptors and kept weights of the chunk
    if (g < p.G) {
        if (lane < ckv) cp_async8(s_desc + lane, p.desc + (size_t)g * p.C + c0 + lane);
        const uint32_t beg = s_kb[warp * kMaxBoundaries + k], end = s_kb[warp * kMaxBoundaries + k + 1];
        for (uint32_t i = beg + lane; i < end; i += 32) cp_async16(s_vals + (i - beg), p.vals + i);
    }
}

template <int S, int RY, int RX, typename TIn>
__global__ void __launch_bounds__(kThreads, 1) pconv_main(const MainParams p) {
    constexpr int WY = Win<S, RY, RX>::WY, WX = Win<S, RY, RX>::WX;
    constexpr int NST = 3;
    extern __shared__ __align__(16) unsigned char smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // CTA -> (spatial tile, filter chunk); filter chunk fastest so CTAs sharing a tile run together
    const int cta = blockIdx.x;
    const int fchunk = cta % p.n_fchunks;
    int t = cta / p.n_fchunks;
    const int tx = t % p.tiles_x;
    t /= p.tiles_x;
    const int ty = t % p.tiles_y;
    const int tn = t / p.tiles_y;
    const int n0 = tn * p.NB;
    const int oy0 = ty * p.BY * RY, ox0 = tx * p.BX * RX;
    const int iy0 = oy0 * S - 1, ix0 = ox0 * S - 1;
    const int g = fchunk * kWarps + warp;

    // shared memory carve-up
    const int vals_per_warp = kF * p.CK;
    float* s_in = reinterpret_cast<float*>(smem);
    float4* s_vals = reinterpret_cast<float4*>(s_in + (size_t)NST * p.stage_floats);
    uint64_t* s_desc = reinterpret_cast<uint64_t*>(s_vals + (size_t)NST * kWarps * vals_per_warp);
    uint32_t* s_kb = reinterpret_cast<uint32_t*>(s_desc + (size_t)NST * kWarps * p.CK);

    // chunk boundaries of this warp's group in the kept-weight stream
    if (g < p.G) {
        for (int i = lane; i <= p.n_chunks; i += 32)
            s_kb[warp * kMaxBoundaries + i] = p.kofs[(size_t)g * p.C + min(i * p.CK, p.C)];
    }
    __syncthreads();

    // lane -> block
    const int blk = lane;
    const int per_img = p.BY * p.BX;
    const int img = blk / per_img;
    const int by = (blk % per_img) / p.BX, bx = blk % p.BX;
    const bool active = img < p.NB;
    const int lane_off = active ? (img * p.IH + by * RY * S) * p.pitch + bx * RX * S : 0;
    const int plane = p.NB * p.IH * p.pitch;

    float acc[kF][RY * RX];
#pragma unroll
    for (int f = 0; f < kF; ++f)
#pragma unroll
        for (int i = 0; i < RY * RX; ++i) acc[f][i] = 0.0f;

#pragma unroll
    for (int s = 0; s < NST - 1; ++s) {
        if (s < p.n_chunks)
            stage_chunk<TIn>(p, s, s_in + (size_t)s * p.stage_floats, s_desc + (size_t)(s * kWarps + warp) * p.CK,
                             s_vals + (size_t)(s * kWarps + warp) * vals_per_warp, s_kb, g, n0, iy0, ix0);
        cp_commit();
    }

    for (int k = 0; k < p.n_chunks; ++k) {
        cp_wait<NST - 2>();
        __syncthreads();
        {
            const int kn = k + NST - 1, sb = kn % NST;
            if (kn < p.n_chunks)
                stage_chunk<TIn>(p, kn, s_in + (size_t)sb * p.stage_floats,
                                 s_desc + (size_t)(sb * kWarps + warp) * p.CK,
                                 s_vals + (size_t)(sb * kWarps + warp) * vals_per_warp, s_kb, g, n0, iy0, ix0);
            cp_commit();
        }
        if (g >= p.G) continue;
        const int sb = k % NST;
        const float* s_base = s_in + (size_t)sb * p.stage_floats + lane_off;
        const uint64_t* sd = s_desc + (size_t)(sb * kWarps + warp) * p.CK;
        const float4* sv = s_vals + (size_t)(sb * kWarps + warp) * vals_per_warp;
        const int ckv = min(p.CK, p.C - k * p.CK);
        int voff = 0;
        for (int cl = 0; cl < ckv; ++cl) {
            uint64_t d = sd[cl];
            const int cnt = (int)(d & 15u);
            if (cnt == 0) continue;
            d >>= 4;
            float win[WY][WX];
            const float* wp = s_base + (size_t)cl * plane;
#pragma unroll
            for (int r = 0; r < WY; ++r) {
#pragma unroll
                for (int c = 0; c < WX; c += 4) {
                    if (c + 4 <= WX) {
                        const float4 v = *reinterpret_cast<const float4*>(wp + r * p.pitch + c);
                        win[r][c] = v.x;
                        win[r][c + 1] = v.y;
                        win[r][c + 2] = v.z;
                        win[r][c + 3] = v.w;
                    } else if (c + 2 <= WX) {
                        const float2 v = *reinterpret_cast<const float2*>(wp + r * p.pitch + c);
                        win[r][c] = v.x;
                        win[r][c + 1] = v.y;
                        if (c + 3 <= WX) win[r][c + 2] = wp[r * p.pitch + c + 2];
                    } else {
                        win[r][c] = wp[r * p.pitch + c];
                    }
                }
            }
            for (int j = 0; j < cnt; ++j) {
                const float4 w = sv[voff + j];
                const int code = (int)(d & 63u);
                d >>= 6;
                dispatch<S, RY, RX, WY, WX>(code, w, acc, win);
            }
            voff += cnt;
        }
    }
    cp_wait<0>();

    // epilogue: bias + ReLU + store to the original channel of every slot
    if (g >= p.G || !active) return;
    const int n = n0 + img;
    if (n >= p.N) return;
    const int oyb = oy0 + by * RY, oxb = ox0 + bx * RX;
    using TOut = TIn;
    TOut* y = static_cast<TOut*>(p.y);
#pragma unroll
    for (int f = 0; f < kF; ++f) {
        const uint32_t co = p.perm[g * kF + f];
        if (co == kPadSlot) continue;
        const float b = p.bias ? p.bias[co] : 0.0f;
        TOut* yc = y + ((size_t)n * p.Cout + co) * p.Ho * p.Wo;
#pragma unroll
        for (int r = 0; r < RY; ++r) {
            const int oy = oyb + r;
            if (oy >= p.Ho) break;
            TOut* yr = yc + (size_t)oy * p.Wo;
            float v[RX];
#pragma unroll
            for (int c = 0; c < RX; ++c) {
                float a = acc[f][r * RX + c] + b;
                v[c] = p.relu ? fmaxf(a, 0.0f) : a;
            }
            if (RX == 4 && p.vec_store && oxb + RX <= p.Wo) {
                if constexpr (sizeof(TOut) == 4) {
                    *reinterpret_cast<float4*>(yr + oxb) = make_float4(v[0], v[1], v[2], v[3]);
                } else {
                    __half2 h0 = __floats2half2_rn(v[0], v[1]);
                    __half2 h1 = __floats2half2_rn(v[2], v[3]);
                    uint2 u;
                    u.x = *reinterpret_cast<unsigned*>(&h0);
                    u.y = *reinterpret_cast<unsigned*>(&h1);
                    *reinterpret_cast<uint2*>(yr + oxb) = u;
                }
            } else {
#pragma unroll
                for (int c = 0; c < RX; ++c)
                    if (oxb + c < p.Wo) yr[oxb + c] = from_f32<TOut>(v[c]);
            }
        }
    }
}

// ------------------------------------------------------------------------------ depthwise

// One warp per (image, slot): channel co = perm[slot] convolves its own plane with its one
// pattern (warp-uniform, compile-time taps).  Each lane produces outputs strided by 32.
template <int S, int P_, typename T>
__device__ __forceinline__ void dw_plane(const T* xp, T* yp, int H, int W, int Ho, int Wo, float4 w,
                                         float b, int relu, int lane) {
    constexpr int t0 = ktap(P_, 0), t1 = ktap(P_, 1), t2 = ktap(P_, 2), t3 = ktap(P_, 3);
    const float wv[4] = {w.x, w.y, w.z, w.w};
    constexpr int tt[4] = {t0, t1, t2, t3};
    const int total = Ho * Wo;
    for (int o = lane; o < total; o += 32) {
        const int oy = o / Wo, ox = o % Wo;
        float a = 0.0f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int iy = oy * S + tt[k] / 3 - 1, ix = ox * S + tt[k] % 3 - 1;
            if (iy >= 0 && iy < H && ix >= 0 && ix < W) a = fmaf(wv[k], to_f32<T>(xp[(size_t)iy * W + ix]), a);
        }
        a += b;
        yp[o] = from_f32<T>(relu ? fmaxf(a, 0.0f) : a);
    }
}

template <int S, typename T>
__global__ void __launch_bounds__(256) pconv_depthwise(const T* __restrict__ x, T* __restrict__ y,
                                                       const float* __restrict__ bias, const uint32_t* perm,
                                                       const uint64_t* desc, const uint32_t* kofs,
                                                       const float4* vals, int C, int H, int W, int Ho,
                                                       int Wo, int G, int relu) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.x % G, n = blockIdx.x / G;
    const int slot = g * kF + warp;
    const uint32_t co = perm[slot];
    if (co == kPadSlot) return;
    uint64_t d = desc[g];
    const int cnt = (int)(d & 15u);
    d >>= 4;
    int pat = -1, j = 0;
    for (int e = 0; e < cnt; ++e) {
        const int code = (int)((d >> (6 * e)) & 63u);
        if ((code >> 3) == warp) { pat = code & 7; j = e; }
    }
    const float b = bias ? bias[co] : 0.0f;
    const T* xp = x + ((size_t)n * C + co) * H * W;
    T* yp = y + ((size_t)n * C + co) * Ho * Wo;
    if (pat < 0) {   // pruned kernel: the output is sigma(bias)
        const float v = relu ? fmaxf(b, 0.0f) : b;
        for (int o = lane; o < Ho * Wo; o += 32) yp[o] = from_f32<T>(v);
        return;
    }
    const float4 w = vals[kofs[g] + j];
    switch (pat) {
        case 0: dw_plane<S, 0, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        case 1: dw_plane<S, 1, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        case 2: dw_plane<S, 2, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        case 3: dw_plane<S, 3, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        case 4: dw_plane<S, 4, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        case 5: dw_plane<S, 5, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        case 6: dw_plane<S, 6, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
        default: dw_plane<S, 7, T>(xp, yp, H, W, Ho, Wo, w, b, relu, lane); break;
    }
}

// ------------------------------------------------------------------------------ generic path

struct TapTable {
    int8_t t[kMaxPatterns][4];
};

// Any pattern library: one thread per output, taps read from a table (slow, for libraries other
// than the compiled one).  Dense or depthwise (cin_g == 1 and ci == co).
template <typename T>
__global__ void pconv_generic(const T* __restrict__ x, T* __restrict__ y, const float* __restrict__ bias,
                              const uint32_t* perm, const uint64_t* desc, const uint32_t* kofs,
                              const float4* vals, TapTable taps, int N, int C, int cin_g, int dw, int H,
                              int W, int Cout, int Ho, int Wo, int S, int relu) {
    const long long total = (long long)N * Cout * Ho * Wo;
    for (long long o = blockIdx.x * (long long)blockDim.x + threadIdx.x; o < total;
         o += (long long)gridDim.x * blockDim.x) {
        const int ox = (int)(o % Wo);
        long long r = o / Wo;
        const int oy = (int)(r % Ho);
        r /= Ho;
        const int slot = (int)(r % Cout);
        const int n = (int)(r / Cout);
        const uint32_t co = perm[slot];
        const int g = slot / kF, f = slot % kF;
        float a = 0.0f;
        for (int ci = 0; ci < cin_g; ++ci) {
            uint64_t d = desc[(size_t)g * cin_g + ci];
            const int cnt = (int)(d & 15u);
            d >>= 4;
            for (int e = 0; e < cnt; ++e) {
                const int code = (int)((d >> (6 * e)) & 63u);
                if ((code >> 3) != f) continue;
                const int pat = code & 7;
                const float4 w = vals[kofs[(size_t)g * cin_g + ci] + e];
                const float wv[4] = {w.x, w.y, w.z, w.w};
                const int xc = dw ? (int)co : ci;
                for (int k = 0; k < 4; ++k) {
                    const int tp = taps.t[pat][k];
                    const int iy = oy * S + tp / 3 - 1, ix = ox * S + tp % 3 - 1;
                    if (iy >= 0 && iy < H && ix >= 0 && ix < W)
                        a = fmaf(wv[k], to_f32<T>(x[(((size_t)n * C + xc) * H + iy) * W + ix]), a);
                }
            }
        }
        a += bias ? bias[co] : 0.0f;
        y[(((size_t)n * Cout + co) * Ho + oy) * Wo + ox] = from_f32<T>(relu ? fmaxf(a, 0.0f) : a);
    }
}

// ------------------------------------------------------------------------------ max-pool

template <typename T>
__global__ void maxpool2x2(const T* __restrict__ x, T* __restrict__ y, long long planes, int H, int W) {
    const int Ho = H / 2, Wo = W / 2;
    const long long total = planes * Ho * Wo;
    for (long long o = blockIdx.x * (long long)blockDim.x + threadIdx.x; o < total;
         o += (long long)gridDim.x * blockDim.x) {
        const int ox = (int)(o % Wo);
        const long long r = o / Wo;
        const int oy = (int)(r % Ho);
        const long long pl = r / Ho;
        const T* xp = x + (pl * H + 2 * oy) * W + 2 * ox;
        const float a = fmaxf(to_f32<T>(xp[0]), to_f32<T>(xp[1]));
        const float b = fmaxf(to_f32<T>(xp[W]), to_f32<T>(xp[W + 1]));
        y[o] = from_f32<T>(fmaxf(a, b));
    }
}

// ------------------------------------------------------------------------------ host side

int sm_count() {
    static std::atomic<int> cached[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    if (dev < 64 && cached[dev].load() > 0) return cached[dev].load();
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    if (dev < 64) cached[dev].store(n);
    return n;
}

struct Tile {
    int BY, BX, NB;
};

// Spatial tile of 32 lane-blocks that minimises the number of CTA waves, then wasted lanes.
Tile choose_tile(int N, int Ho, int Wo, int RY, int RX, int n_fchunks) {
    const int nby = (Ho + RY - 1) / RY, nbx = (Wo + RX - 1) / RX;
    const long long slots = sm_count();
    Tile best{1, 1, 1};
    long long best_waves = LLONG_MAX, best_cover = LLONG_MAX;
    int best_bx = 0;
    for (int bx = 1; bx <= std::min(nbx, 32); ++bx) {
        for (int by = 1; by <= std::min(nby, 32 / bx); ++by) {
            const int nb = std::max(1, std::min(N, 32 / (bx * by)));
            const long long tiles = (long long)((N + nb - 1) / nb) * ((nby + by - 1) / by) * ((nbx + bx - 1) / bx);
            const long long ctas = tiles * n_fchunks;
            const long long waves = (ctas + slots - 1) / slots;
            const long long cover = tiles * 32;   // lanes issued
            if (waves < best_waves || (waves == best_waves && (cover < best_cover ||
                                                               (cover == best_cover && bx > best_bx)))) {
                best = Tile{by, bx, nb};
                best_waves = waves;
                best_cover = cover;
                best_bx = bx;
            }
        }
    }
    return best;
}

template <int S, int RY, int RX, typename T>
int launch_main(const pp_layer* L, const void* x, void* y, const float* bias, int relu, int N, int H, int W,
                int Ho, int Wo, cudaStream_t st) {
    MainParams p{};
    p.x = x;
    p.y = y;
    p.bias = bias;
    const unsigned char* img = static_cast<const unsigned char*>(L->dev);
    p.perm = reinterpret_cast<const uint32_t*>(img + L->off_perm);
    p.desc = reinterpret_cast<const uint64_t*>(img + L->off_desc);
    p.kofs = reinterpret_cast<const uint32_t*>(img + L->off_kofs);
    p.vals = reinterpret_cast<const float4*>(img + L->off_vals);
    p.N = N;
    p.C = L->cin_g;
    p.H = H;
    p.W = W;
    p.Cout = L->cout;
    p.Ho = Ho;
    p.Wo = Wo;
    p.G = L->G;
    p.relu = relu;
    p.n_fchunks = (L->G + kWarps - 1) / kWarps;
    const Tile t = choose_tile(N, Ho, Wo, RY, RX, p.n_fchunks);
    p.BY = t.BY;
    p.BX = t.BX;
    p.NB = t.NB;
    p.tiles_x = ((Wo + RX - 1) / RX + t.BX - 1) / t.BX;
    p.tiles_y = ((Ho + RY - 1) / RY + t.BY - 1) / t.BY;
    p.tiles_n = (N + t.NB - 1) / t.NB;
    p.IH = (t.BY * RY - 1) * S + 3;
    p.IW = (t.BX * RX - 1) * S + 3;
    p.pitch = (p.IW + 3) / 4 * 4;
    // channels per stage: fill ~40 KB of input per stage, at most 32, at least 1
    const int per_ci = p.NB * p.IH * p.pitch;
    int ck = std::max(1, std::min(32, (40 * 1024 / 4) / std::max(per_ci, 1)));
    ck = std::min(ck, L->cin_g);
    p.n_chunks = (L->cin_g + ck - 1) / ck;
    if (p.n_chunks + 1 > kMaxBoundaries) {
        ck = (L->cin_g + kMaxBoundaries - 2) / (kMaxBoundaries - 1);
        p.n_chunks = (L->cin_g + ck - 1) / ck;
    }
    constexpr int NST = 3;
    auto smem_bytes = [&](int c) {
        return (size_t)NST * c * per_ci * 4 + (size_t)NST * kWarps * kF * c * 16 + (size_t)NST * kWarps * c * 8 +
               (size_t)kWarps * kMaxBoundaries * 4;
    };
    while (ck > 1 && smem_bytes(ck) > 200 * 1024) --ck;
    p.n_chunks = (L->cin_g + ck - 1) / ck;
    if (p.n_chunks + 1 > kMaxBoundaries) return PP_ERR_SHAPE;
    p.CK = ck;
    p.stage_floats = ck * per_ci;
    p.vec_store = (RX == 4) && (Wo % 4 == 0) &&
                  ((reinterpret_cast<uintptr_t>(y) % (4 * sizeof(T))) == 0);
    const size_t smem = smem_bytes(ck);
    if (smem > 227 * 1024) return PP_ERR_SHAPE;
    auto kern = pconv_main<S, RY, RX, T>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return PP_ERR_CUDA;
    const long long ctas = (long long)p.tiles_n * p.tiles_y * p.tiles_x * p.n_fchunks;
    if (ctas > INT_MAX) return PP_ERR_SHAPE;
    kern<<<(unsigned)ctas, kThreads, smem, st>>>(p);
    return cudaGetLastError() == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

template <typename T>
int launch_depthwise(const pp_layer* L, const void* x, void* y, const float* bias, int relu, int N, int H, int W,
                     int Ho, int Wo, cudaStream_t st) {
    const unsigned char* img = static_cast<const unsigned char*>(L->dev);
    const auto* perm = reinterpret_cast<const uint32_t*>(img + L->off_perm);
    const auto* desc = reinterpret_cast<const uint64_t*>(img + L->off_desc);
    const auto* kofs = reinterpret_cast<const uint32_t*>(img + L->off_kofs);
    const auto* vals = reinterpret_cast<const float4*>(img + L->off_vals);
    const long long blocks = (long long)N * L->G;
    if (blocks > INT_MAX) return PP_ERR_SHAPE;
    if (L->stride == 1)
        pconv_depthwise<1, T><<<(unsigned)blocks, 256, 0, st>>>(static_cast<const T*>(x), static_cast<T*>(y), bias,
                                                                 perm, desc, kofs, vals, L->cout, H, W, Ho, Wo,
                                                                 L->G, relu);
    else
        pconv_depthwise<2, T><<<(unsigned)blocks, 256, 0, st>>>(static_cast<const T*>(x), static_cast<T*>(y), bias,
                                                                 perm, desc, kofs, vals, L->cout, H, W, Ho, Wo,
                                                                 L->G, relu);
    return cudaGetLastError() == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

template <typename T>
int launch_generic(const pp_layer* L, const void* x, void* y, const float* bias, int relu, int N, int H, int W,
                   int Ho, int Wo, cudaStream_t st) {
    const unsigned char* img = static_cast<const unsigned char*>(L->dev);
    TapTable tt{};
    for (int p = 0; p < L->n_patterns; ++p) {
        int n = 0;
        for (int t = 0; t < 9; ++t)
            if ((L->masks[p] >> t) & 1u) tt.t[p][n++] = (int8_t)t;
    }
    const long long total = (long long)N * L->cout * Ho * Wo;
    const int blocks = (int)std::min<long long>((total + 255) / 256, (long long)sm_count() * 32);
    pconv_generic<T><<<std::max(blocks, 1), 256, 0, st>>>(
        static_cast<const T*>(x), static_cast<T*>(y), bias, reinterpret_cast<const uint32_t*>(img + L->off_perm),
        reinterpret_cast<const uint64_t*>(img + L->off_desc), reinterpret_cast<const uint32_t*>(img + L->off_kofs),
        reinterpret_cast<const float4*>(img + L->off_vals), tt, N, L->depthwise ? L->cout : L->cin_g, L->cin_g,
        L->depthwise ? 1 : 0, H, W, L->cout, Ho, Wo, L->stride, relu);
    return cudaGetLastError() == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    const uintptr_t x0 = reinterpret_cast<uintptr_t>(a), y0 = reinterpret_cast<uintptr_t>(b);
    return x0 < y0 + nb && y0 < x0 + na;
}

}  // namespace

extern "C" {

int pp_bind_device(pp_handle h, void* dev_image, size_t bytes, void* stream) {
    if (!h || !dev_image) return PP_ERR_NULL;
    if (bytes < h->image.size()) return PP_ERR_BUFFER;
    if (reinterpret_cast<uintptr_t>(dev_image) % 256 != 0) return PP_ERR_ALIGN;
    if (cudaMemcpyAsync(dev_image, h->image.data(), h->image.size(), cudaMemcpyHostToDevice,
                        static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return PP_ERR_CUDA;
    h->dev = dev_image;
    h->dev_bytes = bytes;
    return PP_OK;
}

int pp_conv(pp_handle h, const void* x, int dtype, int N, int H, int W, const float* bias, int relu, void* y,
            void* stream) {
    if (!h) return PP_ERR_NULL;
    if (!h->dev) return PP_ERR_NOT_BOUND;
    if (dtype != PP_F32 && dtype != PP_F16) return PP_ERR_DTYPE;
    if (N < 0 || H < 1 || W < 1) return PP_ERR_SHAPE;
    if (relu != 0 && relu != 1) return PP_ERR_ARG;
    if (N == 0) return PP_OK;
    if (!x || !y) return PP_ERR_NULL;
    const int C = h->depthwise ? h->cout : h->cin_g;
    const int Ho = (H - 1) / h->stride + 1, Wo = (W - 1) / h->stride + 1;
    const size_t es = dtype == PP_F32 ? 4 : 2;
    const size_t xb = (size_t)N * C * H * W * es, yb = (size_t)N * h->cout * Ho * Wo * es;
    if ((size_t)N * C * H * W >= (1ull << 40) || (size_t)N * h->cout * Ho * Wo >= (1ull << 40)) return PP_ERR_SHAPE;
    if (reinterpret_cast<uintptr_t>(x) % es || reinterpret_cast<uintptr_t>(y) % es) return PP_ERR_ALIGN;
    if (bias && reinterpret_cast<uintptr_t>(bias) % 4) return PP_ERR_ALIGN;
    if (overlaps(x, xb, y, yb)) return PP_ERR_BUFFER;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const bool f16 = dtype == PP_F16;
    if (!h->fast) {
        return f16 ? launch_generic<__half>(h, x, y, bias, relu, N, H, W, Ho, Wo, st)
                   : launch_generic<float>(h, x, y, bias, relu, N, H, W, Ho, Wo, st);
    }
    if (h->depthwise) {
        return f16 ? launch_depthwise<__half>(h, x, y, bias, relu, N, H, W, Ho, Wo, st)
                   : launch_depthwise<float>(h, x, y, bias, relu, N, H, W, Ho, Wo, st);
    }
    if (h->stride == 1)
        return f16 ? launch_main<1, 4, 4, __half>(h, x, y, bias, relu, N, H, W, Ho, Wo, st)
                   : launch_main<1, 4, 4, float>(h, x, y, bias, relu, N, H, W, Ho, Wo, st);
    return f16 ? launch_main<2, 2, 4, __half>(h, x, y, bias, relu, N, H, W, Ho, Wo, st)
               : launch_main<2, 2, 4, float>(h, x, y, bias, relu, N, H, W, Ho, Wo, st);
}

int pp_maxpool2x2(const void* x, int dtype, int N, int C, int H, int W, void* y, void* stream) {
    if (dtype != PP_F32 && dtype != PP_F16) return PP_ERR_DTYPE;
    if (N < 0 || C < 1 || H < 2 || W < 2) return PP_ERR_SHAPE;
    if (N == 0) return PP_OK;
    if (!x || !y) return PP_ERR_NULL;
    const size_t es = dtype == PP_F32 ? 4 : 2;
    if (reinterpret_cast<uintptr_t>(x) % es || reinterpret_cast<uintptr_t>(y) % es) return PP_ERR_ALIGN;
    const long long planes = (long long)N * C;
    if (overlaps(x, (size_t)planes * H * W * es, y, (size_t)planes * (H / 2) * (W / 2) * es)) return PP_ERR_BUFFER;
    const long long total = planes * (H / 2) * (W / 2);
    const int blocks = (int)std::max<long long>(1, std::min<long long>((total + 255) / 256, (long long)sm_count() * 64));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (dtype == PP_F32)
        maxpool2x2<float><<<blocks, 256, 0, st>>>(static_cast<const float*>(x), static_cast<float*>(y), planes, H, W);
    else
        maxpool2x2<__half><<<blocks, 256, 0, st>>>(static_cast<const __half*>(x), static_cast<__half*>(y), planes, H, W);
    return cudaGetLastError() == cudaSuccess ? PP_OK : PP_ERR_CUDA;
}

}  // extern "C"
