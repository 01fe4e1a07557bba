/*
 * patconv.h -- C ABI of libpatconv: pattern-pruned 3x3 convolution inference on one GB300.
 *
 * Method (arXiv 2003.06513):
 *   - kernel pattern pruning (§3.2): every kept 3x3 kernel keeps exactly 4 weights whose
 *     positions form one pattern of a small library P = {M_1..M_m} (§4.2, m = 6..8);
 *   - the projection onto that constraint set keeps, per kernel, the pattern whose pruned kernel
 *     has the largest Frobenius norm (§4.3, Eq. 5-6);
 *   - connectivity pruning (§4.4) keeps at most beta kernels per layer;
 *   - the compiler-level passes (§3.4) group filters of similar pattern sequence ("filter kernel
 *     reorder") and store the kept weights compactly ("compressed weight storage");
 *   - the layer computes X_n = sigma(W_n X_{n-1} + b_n) (§4.1, Eq. 1) with sigma = ReLU or
 *     identity, as a 3x3 convolution with zero padding 1.
 *
 * Conventions shared by every entry point:
 *   - every function returns a pp_status (0 = PP_OK, negative = error); no exception, abort or
 *     device synchronisation crosses the ABI; out-parameters are written only on PP_OK;
 *   - the library owns host memory only (the handle).  Device memory and streams belong to the
 *     caller; streams are passed as `void*` holding a cudaStream_t (NULL = legacy default);
 *   - taps are numbered in raster order t = 3*(dy+1) + (dx+1), dy, dx in {-1,0,1}; a pattern is
 *     a 9-bit mask with bit t set for each kept tap;
 *   - tensors are contiguous NCHW; weights are host fp32 [Cout][Cin/groups][3][3];
 *   - kernels are launched with programmatic dependent launch on a stream that is not being
 *     captured into a CUDA graph (the streamed depthwise kernel also under capture): a
 *     convolution may start its set-up (reading the layer's bound device image) while the kernel
 *     before it on the stream finishes, and reads or writes no activation and reads no bias
 *     before that kernel has completed, so stream order holds as for a plain launch.  The
 *     environment variable PATCONV_PDL=0 (read once) makes every launch a plain one.
 *
 * Thread safety: a handle is immutable after pp_pack/pp_bind_device, so pp_conv on one handle
 * may be called from several host threads and streams at once.
 */
#ifndef PATCONV_H
#define PATCONV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pp_layer* pp_handle;

typedef enum {
    PP_OK = 0,
    PP_ERR_NULL = -1,         /* a required pointer is NULL                                  */
    PP_ERR_SHAPE = -2,        /* a size is out of range or inconsistent                      */
    PP_ERR_PATTERN = -3,      /* pattern library invalid (count, popcount, duplicates)       */
    PP_ERR_KEEP = -4,         /* keep ratio outside (0, 1] or NaN                            */
    PP_ERR_NONFINITE = -5,    /* a weight is NaN or infinite                                 */
    PP_ERR_ALIGN = -6,        /* a device pointer is not aligned as documented               */
    PP_ERR_DTYPE = -7,        /* unknown pp_dtype                                            */
    PP_ERR_NOT_BOUND = -8,    /* pp_conv before pp_bind_device                               */
    PP_ERR_BUFFER = -9,       /* caller buffer too small / wrong size, or x and y overlap     */
    PP_ERR_CUDA = -10,        /* a CUDA runtime call failed (launch or copy)                 */
    PP_ERR_ARG = -11,         /* any other invalid argument (section, query key, flag)       */
    PP_ERR_ALLOC = -12,       /* host allocation failed                                      */
    PP_ERR_SCRATCH = -13,     /* pp_conv_static_scratch: the call needs more scratch than the
                                 static array holds                                           */
    PP_ERR_PATH = -14         /* the layer's kernel does not offer the requested fusion        */
} pp_status;

typedef enum { PP_F32 = 0, PP_F16 = 1 } pp_dtype;

/* Sections of a packed layer (pp_export).  Byte layouts:
 *   HEADER u32[16]: 'PPK1' (0x314B5050), version 1, Cout, Cin_g, groups, stride, n_patterns,
 *                   beta, F (= 8), G = ceil(Cout/8), masks two per word (low half first), 0, 0
 *   PID    i8 [Cout][Cin_g]   pattern index of each kernel, -1 = pruned (original order)
 *   PERM   u32[G*8]           original filter of each slot, 0xFFFFFFFF = padding slot
 *   DESC   u64[G][Cin_g]      bits 0-3: kept kernels c of group g at input channel ci; entry
 *                             j < c at bits 4+6j..9+6j = (slot << 3) | pattern, slots ascending
 *   KOFS   u32[G*Cin_g + 1]   kept kernels before (g, ci) in (g, ci, slot) order; last = beta
 *   VALS   f32[beta][4]       kept weights in (g, ci, slot) order, taps ascending (bit copies)
 *   DENSE  f32[Cout][Cin_g][9] projected weights with zeros in place
 *   IMAGE  the device image: PERM | DESC | KOFS | VALS, each starting at a multiple of 256 B.
 * Filter slot order (filter kernel reorder, §3.4): filters sorted by kept count descending, then
 * by their pattern-index sequence over ci (pruned = 15) ascending, then by original index; the
 * j-th filter of that order takes slot r = j / G of group g = j % G (g = G-1 - j % G when r is
 * odd), so every group holds a similar number of kept kernels. */
typedef enum {
    PP_SEC_HEADER = 0, PP_SEC_PID = 1, PP_SEC_PERM = 2, PP_SEC_DESC = 3,
    PP_SEC_KOFS = 4, PP_SEC_VALS = 5, PP_SEC_DENSE = 6, PP_SEC_IMAGE = 7
} pp_section;

typedef enum {
    PP_Q_BETA = 0, PP_Q_COUT = 1, PP_Q_CIN_G = 2, PP_Q_GROUPS = 3, PP_Q_STRIDE = 4,
    PP_Q_N_GROUPS = 5, PP_Q_N_PATTERNS = 6, PP_Q_IMAGE_BYTES = 7,
    PP_Q_FAST_PATH = 8,       /* 1 if the library equals pp_default_patterns (compiled bodies)  */
    PP_Q_SECTION_BYTES = 16   /* + section id: byte size of that section                      */
} pp_query_key;

/* The 8-pattern library the fast kernels are compiled for (§3.2, §4.2): indices 0-3 keep the
 * centre and three of the four edge neighbours (dropping up, left, right, down in turn);
 * indices 4-7 keep the centre, one edge neighbour (up, left, right, down) and the two corners
 * flanking it.  Writes min(capacity, 8) masks to `masks` and returns 8 (or a negative status
 * if masks is NULL with capacity > 0). */
int pp_default_patterns(uint16_t* masks, int capacity);

/* Pattern-library design heuristic (§4.2): the central weight is always kept, and each kernel
 * proposes the pattern made of the centre and its three largest non-central weights (largest
 * magnitude; equal magnitudes take the lower raster tap first); the m most frequent proposals
 * over all kernels given form the library, ordered by frequency (descending), equal counts by
 * mask value (ascending) -- the order matters, because projection ties go to the lower index.
 *   W       HOST fp32 [n_kernels][9]: every 3x3 kernel of the network (or layer), raster taps;
 *   m       library size, 1..8 (§4.2 finds 6-8 best);
 *   masks   HOST out, room for m masks; *n_masks gets the number written (fewer than m when
 *           fewer distinct proposals exist).
 * A library other than pp_default_patterns packs and runs through pp_pack / pp_conv like the
 * default one; dense layers then take the generic kernel (taps from a table, slower).
 * Errors: PP_ERR_NULL, PP_ERR_SHAPE (n_kernels == 0, m outside 1..8), PP_ERR_NONFINITE. */
int pp_design_patterns(const float* W, size_t n_kernels, int m, uint16_t* masks, int* n_masks);

/* Pattern projection (§4.3 Eq. 6), connectivity pruning (§4.4) and packing (§3.4) of one layer.
 *   W        host fp32 [Cout][Cin/groups][3][3], read only, caller-owned;
 *   groups   1 (dense) or Cout == Cin (depthwise);
 *   stride   1 or 2 (padding is always 1);
 *   masks    n_patterns 9-bit masks, 1 <= n_patterns <= 8, each with exactly 4 bits, distinct;
 *   keep     connectivity keep ratio in (0, 1]: beta = floor(keep * Cout * Cin_g + 0.5) in
 *            float64, clamped to [1, Cout*Cin_g]; the beta kernels with the largest retained
 *            energy survive, ties to the lower flat index co*Cin_g + ci;
 * Projection scores are float64 sums ((a^2 + b^2) + c^2) + d^2 over the pattern's taps in
 * ascending order; ties go to the lowest pattern index.  Host-only: touches no GPU.
 * Errors: PP_ERR_NULL, PP_ERR_SHAPE, PP_ERR_PATTERN, PP_ERR_KEEP, PP_ERR_NONFINITE,
 * PP_ERR_ALLOC.  On success *out owns host memory released by pp_destroy. */
int pp_pack(const float* W, int Cout, int Cin, int groups, int stride,
            const uint16_t* masks, int n_patterns, double keep, pp_handle* out);

/* Read one scalar property (pp_query_key) of a packed layer. */
int pp_query(pp_handle h, int key, int64_t* value);

/* Copy one section (pp_section) into host memory; `bytes` must equal its size exactly
 * (PP_Q_SECTION_BYTES + section), else PP_ERR_BUFFER. */
int pp_export(pp_handle h, int section, void* host_dst, size_t bytes);

/* Upload the device image into caller-owned DEVICE memory `dev_image` (>= PP_Q_IMAGE_BYTES
 * bytes, 256-byte aligned) with an asynchronous host-to-device copy on `stream`, and remember
 * the pointer for pp_conv.  The caller keeps the memory alive (and unmodified) while the handle
 * is used, and must order the copy before the first pp_conv (same stream, or an event).
 * Errors: PP_ERR_NULL, PP_ERR_BUFFER (too small), PP_ERR_ALIGN, PP_ERR_CUDA. */
int pp_bind_device(pp_handle h, void* dev_image, size_t bytes, void* stream);

/* y = sigma(conv3x3(x, W_hat, stride, pad 1) + bias) on the GPU, enqueued on `stream`.
 *   x     DEVICE [N][Cin][H][W] of `dtype` (PP_F32 or PP_F16);
 *   y     DEVICE [N][Cout][Ho][Wo] of the same dtype, Ho = (H-1)/stride + 1 (likewise Wo);
 *         must not overlap x;
 *   bias  DEVICE fp32 [Cout] or NULL (no bias);  relu 0 or 1.
 * Accumulation is fp32 (FFMA on the CUDA cores) in input-channel order; fp16 inputs are
 * widened exactly and the fp16 output is rounded to nearest even.  Pointers need only element
 * alignment; 16-byte aligned x/y with W % 4 == 0 take the vector paths.  N == 0 is a no-op.
 * Validation errors return before any launch; a failed launch returns PP_ERR_CUDA.  Never
 * synchronises. */
int pp_conv(pp_handle h, const void* x, int dtype, int N, int H, int W,
            const float* bias, int relu, void* y, void* stream);

/* pp_conv with an optional caller-owned DEVICE workspace (16-byte aligned, no overlap with x or
 * y).  When one pass over all input channels gives too few CTAs to fill the GPU (small images),
 * the input channels are cut into KS contiguous ranges; each range's CTAs write fp32 partial
 * sums into the workspace ([KS][N][Cout][Ho][Wo]) and a second kernel adds the ranges in order,
 * adds the bias, applies ReLU and rounds to the output type.  The result is deterministic; it
 * can differ from the single-pass sum in the last bits (fp32 summation order).  workspace ==
 * NULL or too small for any split means a single pass.  The dense fast path only; other paths
 * ignore the workspace.  Same errors as pp_conv, plus PP_ERR_ALIGN / PP_ERR_BUFFER for the
 * workspace. */
int pp_conv_ws(pp_handle h, const void* x, int dtype, int N, int H, int W, const float* bias,
               int relu, void* y, void* workspace, size_t workspace_bytes, void* stream);

/* pp_conv_ws followed by a 2x2 max-pool with stride 2, fused into the conv's epilogue: y is
 * DEVICE [N][Cout][Ho/2][Wo/2] (floor: an odd last output row or column is dropped) and holds
 * max over each 2x2 window of sigma(conv + bias).  The forward pass of a layer is sigma(WX + b)
 * (§4.1); the pooling that follows VGG's blocks is the network's, not the paper's method, and is
 * fused here so that the full-resolution map never reaches memory.  Each lane of the kernel owns
 * a 4x4 output block whose origin is even, so every pooling window lies inside one lane.  With a
 * workspace split the partial sums stay full-resolution in the workspace (same size as for
 * pp_conv_ws) and the reduction pools.  Dense layers on the compiled pattern library only
 * (pp_query PP_Q_FAST_PATH == 1); others return PP_ERR_PATH.  Ho and Wo must be at least 2
 * (PP_ERR_SHAPE).  Otherwise the errors of pp_conv_ws. */
int pp_conv_pool_ws(pp_handle h, const void* x, int dtype, int N, int H, int W, const float* bias,
                    int relu, void* y, void* workspace, size_t workspace_bytes, void* stream);

/* Workspace bytes pp_conv_ws would use for this call shape with unlimited workspace (0 when it
 * would not split).  Host-only. */
int pp_conv_workspace_size(pp_handle h, int N, int H, int W, size_t* bytes);

/* Launch plan of pp_conv_ws for a call shape and workspace size, for tests and tuning:
 * info[0] = path (1 dense fast kernel, 2 depthwise kernel, 3 generic kernel); for path 1:
 * info[1] channel splits KS, [2] workspace bytes used, [3] work units (spatial tiles x filter
 * chunks x splits), [4..6] tile BY, BX, NB (4x4 output blocks; NB > 1 images side by side in one
 * stage: whole images, the linear tile's consecutive blocks across images, or bands of BY full
 * block rows where a whole image exceeds the lanes), [7] channels per stage,
 * [8] filter groups and [9] spatial warps per CTA, [10] shared-memory bytes, [11] channel chunks
 * per unit, [12] CTAs launched when the input goes through TMA (fp32 with rows a multiple of 16
 * bytes: persistent CTAs, at most one per SM unless the units overflow a CTA's unit table; the
 * copy fallback launches one CTA per unit), [13] 1 where a stride-1 fp32 launch deals each warp's
 * blocks to its lanes by shared-memory bank group (fewer conflicting window loads; rows of 7 or
 * 14 blocks), else 0; [14] s where the stride-1 blocks of a tile row start at output columns
 * 4j - s instead of 4j: s = 1 (each lane's input window then starts 8 bytes into a 16-byte group,
 * so a window row is one 8-byte and one 16-byte shared load instead of two bank-conflicted 4-byte
 * loads around a 16-byte one; never for pp_conv_pool_ws, whose 2x2 pooling windows must lie
 * inside one block), s = 2 (fp32 pp_conv_pool_ws only: the window starts 4 bytes into a 16-byte
 * group and a row is two 16-byte loads; block origins stay even), else 0; [15] 1 where the launch takes the balanced
 * schedule: one CTA per SM, each taking an equal share of all units' input-channel chunks
 * instead of whole units (whole units leave the SMs of the last partial wave idle); a unit cut
 * between two CTAs is finished by the CTA holding its first chunks, which adds the later ones'
 * raw sums from their workspace slots (workspace: 256 KiB per SM + flags, reported in [2]; the
 * launch is cooperative and resets the flags with a small memset first; the input must go
 * through TMA, or the tile be whole images, else the launch takes whole units), else 0; [16] filter groups per warp (2 for
 * stride-2 layers: 8 warps of 16 filter slots, each input window serving both groups' kept
 * kernels; else 1).  For path 2 (depthwise), assuming
 * x and y 16-byte aligned (else the row-item kernels run): info[1] = 1 streamed kernel in rows
 * mode (bands of whole rows of one plane per tensor copy), 2 streamed kernel in planes mode at
 * stride 2 (one output column per lane), 3 planes mode at stride 1 with rows of even width (two
 * columns per lane), 4 the same for rows of odd width, 5 / 6 tiles mode at stride 1 (each lane a
 * band of 7 output rows by 7 / 14 columns of one plane), 7 tiles mode at stride 2 (a lane a 7x7
 * output plane), 0 the row-item kernels; [3] chunks, [4] output rows per chunk (rows mode) or
 * planes per chunk, [5] shared-memory stages per warp, [6] warps per CTA, [10] shared-memory
 * bytes, [12] CTAs.  Writes min(n_info, 17) values.
 * Host-only. */
int pp_conv_plan(pp_handle h, int N, int H, int W, size_t workspace_bytes, int64_t* info, int n_info);

/* Launch plan of pp_conv_pool_ws (conv with the fused 2x2 max-pool) for a call shape and
 * workspace size: the same fields as pp_conv_plan; info[14] is 0 or 2 here.  Layers without
 * the fused pooling (depthwise, other pattern libraries) return PP_ERR_PATH.  Host-only. */
int pp_conv_pool_plan(pp_handle h, int N, int H, int W, size_t workspace_bytes, int64_t* info,
                      int n_info);

/* The plan of a call with a given dtype (PP_F32, PP_F16) and pool flag (0: pp_conv_ws, 1:
 * pp_conv_pool_ws), fields as pp_conv_plan.  The dtype matters where the planner asks whether
 * the input rows go through TMA (a multiple of 16 bytes), as the balanced schedule needs;
 * pp_conv_plan, pp_conv_pool_plan and pp_conv_workspace_size answer for fp32 calls.  The
 * workspace a call needs is info[2] of the plan with workspace_bytes = SIZE_MAX.  Errors:
 * PP_ERR_DTYPE, PP_ERR_ARG (pool not 0/1), PP_ERR_PATH (pool on a layer without it), and those
 * of pp_conv_plan.  Host-only. */
int pp_conv_plan_dt(pp_handle h, int dtype, int pool, int N, int H, int W, size_t workspace_bytes,
                    int64_t* info, int n_info);

/* pp_conv_ws for callers that cannot allocate device memory (the paper has no counterpart to
 * this entry point).  Some callers are not allowed to call cudaMalloc or any allocating routine:
 * code embedded in a host runtime whose allocator owns all device memory, plugins that must
 * not allocate while serving, or setups where an allocation could block behind other work.
 * Such callers still pass x, y and bias, but get the input-channel split's partial sums in a
 * scratch array that lives in the library itself: a file-scope device array of
 * PP_STATIC_SCRATCH_BYTES (32 MiB) that every GPU loading the library keeps until the process
 * exits.  Nothing is allocated and no allocating routine is called.
 *   - the first call on a device looks up the array's device address (once per device, with
 *     that device current); make that first call before any stream capture;
 *   - the call runs the plan pp_conv_ws would run with an unlimited workspace; where that plan's
 *     split needs more scratch than the array holds (pp_conv_workspace_size reports the need)
 *     it returns PP_ERR_SCRATCH without launching anything, rather than falling back to a plan
 *     that fits.  Such shapes (wide layers on many small images) are rejected here although
 *     pp_conv, which never splits, and pp_conv_ws with a smaller workspace accept them;
 *   - the argument errors of pp_conv_ws (PP_ERR_NULL, _ARG, _ALIGN, _BUFFER, ...) are checked
 *     first and take precedence over PP_ERR_SCRATCH;
 *   - every call on a device shares the one array, which keeps the previous call's contents;
 *     nothing needs clearing (each call writes every partial sum it reads before reading it),
 *     but calls that overlap on the GPU (different streams, or different host threads) race on
 *     it: order them;
 *   - otherwise identical to pp_conv_ws with an unlimited workspace (same plan, same result). */
#define PP_STATIC_SCRATCH_BYTES 33554432
int pp_conv_static_scratch(pp_handle h, const void* x, int dtype, int N, int H, int W,
                           const float* bias, int relu, void* y, void* stream);

/* Size in bytes of the static scratch array behind pp_conv_static_scratch. */
int pp_static_scratch_bytes(size_t* bytes);

/* 2x2 max-pool, stride 2, floor mode: y[n,c,i,j] = max x[n,c,2i+a,2j+b] (a,b in {0,1}).
 * The pooling between VGG blocks; x DEVICE [N][C][H][W], y DEVICE [N][C][H/2][W/2], same dtype,
 * no overlap.  Enqueue only. */
int pp_maxpool2x2(const void* x, int dtype, int N, int C, int H, int W, void* y, void* stream);

/* Device status word of the conv kernels on the current device.  A kernel whose pipeline wait
 * runs out of time (about one second; it never happens in a correct run) records a bit here and
 * returns early instead of hanging: 1 = data stage never arrived, 2 = stage never released,
 * 4 = copies still in flight at exit.  *status gets the word; clear != 0 resets it.  Synchronous
 * (a device-to-host copy); call it between launches, e.g. at the end of a test.
 * Errors: PP_ERR_NULL, PP_ERR_CUDA. */
int pp_device_status(int clear, unsigned int* status);

/* Measured FP32 fused multiply-add peak of the current device in FLOP/s (2 per FMA), the
 * roofline denominator of the dense kernel (the paper has no counterpart): independent
 * fma.rn.f32 chains on every SM, no memory traffic, timed with CUDA events on the legacy default
 * stream, best of `reps` launches of about 2 ms after one warm-up launch.  Synchronous.
 * Errors: PP_ERR_NULL, PP_ERR_ARG (reps outside 1..1000), PP_ERR_CUDA. */
int pp_measure_fp32_peak(int reps, double* flop_per_s);

/* Test hook for the failure path above (the paper has no counterpart): the next launch of the
 * dense pattern-sparse kernel, from any thread, issues none of its input-stage copies and waits
 * only about 10 us for them, so the first pipeline wait of every CTA runs out.  That launch
 * records bit 1 in the status word, writes nothing to y (the call itself returns PP_OK: the
 * failure is on the device) and returns with nothing in flight; the context stays usable and
 * later calls run normally.  One-shot; depthwise and generic kernels ignore it.  Never needed in
 * use.  Returns PP_OK. */
int pp_debug_inject_timeout(void);

/* Release the handle's host memory (the bound device image stays the caller's).  NULL is OK. */
int pp_destroy(pp_handle h);

/* Static English text for a status code. */
const char* pp_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* PATCONV_H */
