#!/usr/bin/env python3
"""Generate pattern_dispatch.h: the channel loop of the pattern-sparse kernel as inline PTX.

One macro per stride, stage type (fp32 stages; fp16 stages, whose window elements are widened to
fp32 as they are loaded) and window alignment processes one pipeline stage (CK input channels)
for one filter group and one lane's 4x4 output block.  Per input channel:

    ld.shared        the group's 64-bit descriptor (count in bits 0-3, then 6-bit
                     (slot << 3 | pattern) codes of the kept kernels, slots ascending)
    ld.shared        the lane's input window, (4-1)*S+3 rows of (4-1)*S+3 elements; row r starts
                     at a register advanced by one channel plane per channel, columns are
                     immediates; stride 2 takes column 0 from the left neighbour lane (a warp
                     shuffle) where that lane holds the block to the left
    per kept kernel:
      ld.shared.v4   its four kept weights (consecutive in the compact storage, §3.4)
      tcgen05.ld     the 16 accumulators of its filter slot from tensor memory
      compare tree   three uniform branches select the body of its pattern
      body           64 fused multiply-adds whose tap operands are compile-time window registers
                     (the four kept positions of the pattern, §3.2): nothing is decoded per element
      tcgen05.st     the accumulators back

Window alignment (stride 1).  The input stage is a tensor copy whose first column sits on a
16-byte boundary, so the output block origin decides where a lane's window column 0 falls:
  * blocks at output columns 4j: column 0 at 3 (mod 4); each row is a 4-byte, a 16-byte and a
    4-byte load, and every lane's 4-byte loads fall on 8 of the 32 banks (4-way conflicts);
  * blocks at output columns 4j - 1 (the "A" macros): column 0 at 2 (mod 4); each row is an
    8-byte load of columns 0-1 and a 16-byte load of columns 2-5, a third fewer shared-memory
    wavefronts and one instruction fewer;
  * blocks at output columns 4j - 2 (the "B" macros, fp32): column 0 at 1 (mod 4); each row is
    two 16-byte loads, of columns -1..2 and 3..6 (the window address is that of column -1), as
    few wavefronts as the "A" layout, and every 2x2 pooling window of the block's outputs stays
    inside the block.
Packed taps.  A tap whose window pairs are the halves of one aligned load runs as fma.rn.f32x2
on pairs of outputs (columns 0-1 and 2-3 of a row; same rounding as two fma.rn.f32): with
blocks at 4j or 4j - 2 the centre-column taps (1, 4, 7), whose pairs are window columns (1, 2)
and (3, 4); with blocks at 4j - 1 the side-column taps (0, 3, 6 and 2, 5, 8), whose pairs are
(0, 1), (2, 3) and (2, 3), (4, 5).  The other taps read pairs that straddle the alignment and
stay scalar.
Taps are applied in ascending raster order for every output.

Two filter groups per warp (the "_G2" macros, stride 2): per input channel both groups'
descriptors are read and the window is loaded once; the kept kernels of the first group, then
those of the second (weights from its own list, accumulators 128 tensor-memory columns up), run
as one visit stream through the same bodies.

Every branch is warp-uniform (bra.uni), so no convergence code surrounds the loop.  The macros'
operands are listed in macro().  The library masks are the eight defaults (centre + 3 of the 4
edge neighbours; centre + one edge + its 2 flanking corners).

Usage: gen_dispatch.py OUT.h
"""
import sys

MASKS = [0x0B8, 0x0B2, 0x09A, 0x03A, 0x017, 0x059, 0x134, 0x1D0]
STRIDES = [1, 2]          # every lane owns a 4x4 output block


def taps(mask):
    return [t for t in range(9) if (mask >> t) & 1]


def macro(S, half=False, shift=0, groups=1, dealt=False):
    RY = RX = 4
    WY, WX = (RY - 1) * S + 3, (RX - 1) * S + 3
    R = RY * RX
    acc = ", ".join(f"a{i}" for i in range(R))
    rows = ", ".join(f"rb{r}" for r in range(WY))
    # operands: %0 channels, %1 descriptor address, %2 weights address, %3 window address of
    # channel 0 (of window column -1 for shift 2), %4 row pitch in bytes, %5 channel plane in
    # bytes, %6 tensor-memory base, %7 nonzero where the left neighbour lane does not hold the
    # block to the left (stride 2); with two filter groups per warp also %8 / %9 the second
    # group's descriptor / weights addresses and %10 nonzero where that group exists (its
    # accumulators sit 128 tensor-memory columns above the first group's)
    packed = S == 1
    aligned = shift == 1
    pairs = (0, 2, 4) if aligned else (1, 3)      # window columns starting an aligned pair

    def packs(dx):                                # tap column dx (0..2) runs as f32x2
        return (dx != 1) if aligned else (dx == 1)
    L = ["{",
         ".reg .pred P, EL;",
         f".reg .b32 cl, cnt, code, ta, pat, va, da, t1, {rows};",
         ".reg .b64 d, dd;",
         f".reg .f32 x<{WY * WX}>, a<{R}>, w<4>, xs<2>;"]
    if packed:   # window pairs xq{5 * row + column}, accumulator pairs, duplicated weights
        L.append(f".reg .b64 xq<{5 * WY}>, ap<{R // 2}>, wq<4>;")
    if half:     # fp16 stage: 16-bit elements widened to fp32 as the window is loaded
        L.append(".reg .b16 h<10>;")
        L.append(".reg .b32 pA, pB, pC, pD;")
    L += [
         "mov.b32 cl, %0;",
         "mov.b32 da, %1;",
         "mov.b32 va, %2;",
         "mov.b32 rb0, %3;",
         "setp.ne.u32 EL, %7, 0;"]
    if groups == 2:
        L[1:1] = [".reg .pred VB;", ".reg .b32 dab, vaa, vab, cb, tot, tb;", ".reg .b64 db;"]
        L += ["mov.b32 dab, %8;", "mov.b32 vab, %9;", "mov.b32 vaa, %2;", "setp.ne.u32 VB, %10, 0;"]
    for r in range(1, WY):
        L.append(f"add.u32 rb{r}, rb{r - 1}, %4;")
    L += ["CL:",
          "setp.eq.u32 P, cl, 0;",
          "@P bra.uni CD;",
          "ld.shared.u64 d, [da];",
          "add.u32 da, da, 8;",
          "cvt.u32.u64 cnt, d;",
          "and.b32 cnt, cnt, 15;"]
    if groups == 2:   # the second group's descriptor (none where the group does not exist)
        L += ["ld.shared.u64 db, [dab];",
              "add.u32 dab, dab, 8;",
              "@!VB mov.b64 db, 0;",
              "cvt.u32.u64 cb, db;",
              "and.b32 cb, cb, 15;",
              "add.u32 tot, cnt, cb;",
              "setp.eq.u32 P, tot, 0;",
              "@P bra.uni CN;"]
    else:
        L += ["setp.eq.u32 P, cnt, 0;",
              "@P bra.uni CN;"]

    def cvt_pair(p, a):                   # two packed halves to x{a}, x{a+1}
        return [f"mov.b32 {{h0, h1}}, {p};", f"cvt.f32.f16 x{a}, h0;", f"cvt.f32.f16 x{a + 1}, h1;"]
    for r in range(WY):
        base = r * WX
        if S == 2 and half:                  # columns 1-8 as two 8-byte loads of four halves
            L.append(f"ld.shared.v2.b32 {{pA, pB}}, [rb{r}+2];")
            L.append(f"ld.shared.v2.b32 {{pC, pD}}, [rb{r}+10];")
            for i, pr in enumerate(("pA", "pB", "pC", "pD")):
                L += cvt_pair(pr, base + 1 + 2 * i)
            L.append(f"shfl.sync.up.b32 x{base}, x{base + 8}, 1, 0, -1;")
            L.append(f"@EL ld.shared.b16 h2, [rb{r}];")
            L.append(f"@EL cvt.f32.f16 x{base}, h2;")
            continue
        if S == 2:
            L.append(f"ld.shared.v4.f32 {{x{base + 1}, x{base + 2}, x{base + 3}, x{base + 4}}}, [rb{r}+4];")
            L.append(f"ld.shared.v4.f32 {{x{base + 5}, x{base + 6}, x{base + 7}, x{base + 8}}}, [rb{r}+20];")
            if dealt:   # blocks dealt to lanes by bank group: the left block's lane is %11
                L.append(f"shfl.sync.idx.b32 x{base}, x{base + 8}, %11, 31, -1;")
            else:
                L.append(f"shfl.sync.up.b32 x{base}, x{base + 8}, 1, 0, -1;")
            L.append(f"@EL ld.shared.f32 x{base}, [rb{r}];")
            continue
        if half and aligned:                 # columns 0-1 (4 bytes), columns 2-5 (8 bytes)
            L.append(f"ld.shared.b32 pA, [rb{r}];")
            L.append(f"ld.shared.v2.b32 {{pB, pC}}, [rb{r}+4];")
            L += cvt_pair("pA", base) + cvt_pair("pB", base + 2) + cvt_pair("pC", base + 4)
        elif half:                           # column 0, columns 1-4 (one 8-byte load), column 5
            L.append(f"ld.shared.b16 h2, [rb{r}];")
            L.append(f"ld.shared.v2.b32 {{pA, pB}}, [rb{r}+2];")
            L.append(f"ld.shared.b16 h3, [rb{r}+10];")
            L.append(f"cvt.f32.f16 x{base}, h2;")
            L += cvt_pair("pA", base + 1) + cvt_pair("pB", base + 3)
            L.append(f"cvt.f32.f16 x{base + 5}, h3;")
        elif shift == 2:                     # columns -1..2 and 3..6 (16 bytes each)
            L.append(f"ld.shared.v4.f32 {{xs0, x{base}, x{base + 1}, x{base + 2}}}, [rb{r}];")
            L.append(f"ld.shared.v4.f32 {{x{base + 3}, x{base + 4}, x{base + 5}, xs1}}, [rb{r}+16];")
        elif aligned:                        # columns 0-1 (8 bytes), columns 2-5 (16 bytes)
            L.append(f"ld.shared.v2.f32 {{x{base}, x{base + 1}}}, [rb{r}];")
            L.append(f"ld.shared.v4.f32 {{x{base + 2}, x{base + 3}, x{base + 4}, x{base + 5}}}, [rb{r}+8];")
        else:                                # column 0, columns 1-4 (16 bytes), column 5
            L.append(f"ld.shared.f32 x{base}, [rb{r}];")
            L.append(f"ld.shared.v4.f32 {{x{base + 1}, x{base + 2}, x{base + 3}, x{base + 4}}}, [rb{r}+4];")
            L.append(f"ld.shared.f32 x{base + 5}, [rb{r}+20];")
        for c0 in pairs:
            L.append(f"mov.b64 xq{5 * r + c0}, {{x{base + c0}, x{base + c0 + 1}}};")
    if groups == 2:
        # one visit stream: the first group's kept kernels (weights from vaa, accumulators at the
        # base), then the second group's (weights from vab, accumulators 128 columns up)
        L += ["shr.b64 dd, d, 4;",
              "mov.b32 va, vaa;",
              "mov.b32 tb, %6;",
              "setp.ne.u32 P, cnt, 0;",
              "@P bra.uni PL;",
              "shr.b64 dd, db, 4;",
              "mov.b32 va, vab;",
              "add.u32 tb, %6, 128;",
              "mov.b32 cnt, cb;"]
        tbase = "tb"
    else:
        L += ["shr.b64 dd, d, 4;"]
        tbase = "%6"
    L += ["PL:",
          "ld.shared.v4.f32 {w0, w1, w2, w3}, [va];",
          "add.u32 va, va, 16;",
          "cvt.u32.u64 code, dd;",
          "shr.b64 dd, dd, 6;",
          "and.b32 pat, code, 7;",
          "and.b32 t1, code, 56;",
          "shl.b32 t1, t1, 1;",
          f"add.u32 ta, {tbase}, t1;",
          f"tcgen05.ld.sync.aligned.32x32b.x{R}.b32 {{{acc}}}, [ta];"]
    if groups == 1:
        L += ["tcgen05.wait::ld.sync.aligned;"]
    L += ["setp.lt.u32 P, pat, 4;", "@P bra.uni T03;",
          "setp.lt.u32 P, pat, 6;", "@P bra.uni T45;",
          "setp.eq.u32 P, pat, 6;", "@P bra.uni B6;", "bra.uni B7;",
          "T45:", "setp.eq.u32 P, pat, 4;", "@P bra.uni B4;", "bra.uni B5;",
          "T03:", "setp.lt.u32 P, pat, 2;", "@P bra.uni T01;",
          "setp.eq.u32 P, pat, 2;", "@P bra.uni B2;", "bra.uni B3;",
          "T01:", "setp.eq.u32 P, pat, 0;", "@P bra.uni B0;", "bra.uni B1;"]
    for p, m in enumerate(MASKS):
        L.append(f"B{p}:")
        if groups == 2:              # the accumulators' load flew during the pattern dispatch
            L.append("tcgen05.wait::ld.sync.aligned;")
        tp = taps(m)
        if packed:
            L += [f"mov.b64 ap{i}, {{a{2 * i}, a{2 * i + 1}}};" for i in range(R // 2)]
            L += [f"mov.b64 wq{k}, {{w{k}, w{k}}};" for k in range(4) if packs(tp[k] % 3)]
        for k in range(4):                   # tap-outer: 16 independent FMAs per tap
            t = tp[k]
            dy, dx = t // 3, t % 3
            if packed and packs(dx):         # outputs (r, 0-1) and (r, 2-3): window pairs of row r + dy
                for r in range(RY):
                    for h in range(2):
                        L.append(f"fma.rn.f32x2 ap{2 * r + h}, wq{k}, xq{5 * (r + dy) + 2 * h + dx}, ap{2 * r + h};")
                continue
            for r in range(RY):
                for c in range(RX):
                    wr = (r * S + dy) * WX + (c * S + dx)
                    o = r * RX + c
                    if packed and c % 2 == 0:
                        L.append(f"mov.b64 {{a{o}, a{o + 1}}}, ap{o // 2};")
                    L.append(f"fma.rn.f32 a{o}, w{k}, x{wr}, a{o};")
                    if packed and c % 2 == 1:
                        L.append(f"mov.b64 ap{o // 2}, {{a{o - 1}, a{o}}};")
        if packed:
            L += [f"mov.b64 {{a{2 * i}, a{2 * i + 1}}}, ap{i};" for i in range(R // 2)]
        if p != len(MASKS) - 1:
            L.append("bra.uni BS;")
    L += ["BS:",
          f"tcgen05.st.sync.aligned.32x32b.x{R}.b32 [ta], {{{acc}}};"]
    if groups == 1:
        L += ["tcgen05.wait::st.sync.aligned;"]
    L += ["sub.u32 cnt, cnt, 1;",
          "setp.ne.u32 P, cnt, 0;",
          "@P bra.uni PL;"]
    if groups == 2:   # first group done: the second group's kept kernels, if any remain
        L += ["setp.ne.u32 P, tb, %6;",
              "@P bra.uni CE;",
              "setp.eq.u32 P, cb, 0;",
              "@P bra.uni CE;",
              "shr.b64 dd, db, 4;",
              "mov.b32 va, vab;",
              "add.u32 tb, %6, 128;",
              "mov.b32 cnt, cb;",
              "bra.uni PL;",
              "CE:",
              "cvt.u32.u64 t1, d;",          # both groups' weight pointers past this channel
              "and.b32 t1, t1, 15;",
              "shl.b32 t1, t1, 4;",
              "add.u32 vaa, vaa, t1;",
              "shl.b32 t1, cb, 4;",
              "add.u32 vab, vab, t1;"]
    L += ["CN:"]
    if groups == 2:   # the channel's stores complete before a later channel loads the same slot
        L += ["tcgen05.wait::st.sync.aligned;"]
    for r in range(WY):
        L.append(f"add.u32 rb{r}, rb{r}, %5;")
    L += ["sub.u32 cl, cl, 1;",
          "bra.uni CL;",
          "CD:",
          "}"]
    body = "\\n\\t".join(L)
    tag = {0: "", 1: "A", 2: "B"}[shift]
    name = f"PP_STAGE_KERNELS_S{S}" + ("_H" if half else "") + ((tag if half else "_" + tag) if tag else "")
    if groups == 2:
        name += "_G2" + ("D" if dealt else "")
        what_g = ", two filter groups per warp" + (", blocks dealt to lanes by bank group" if dealt else "")
    else:
        what_g = ""
    where = {0: "", 1: ", window column 0 at 2 mod 4", 2: ", window column 0 at 1 mod 4"}[shift]
    what = f"stride {S}{', fp16 stage' if half else ''}{where}{what_g}"
    extra_args = ", desc_b, vals_b, valid_b" if groups == 2 else ""
    extra_ops = ', "r"(desc_b), "r"(vals_b), "r"(valid_b)' if groups == 2 else ""
    if dealt:
        extra_args += ", srcl"
        extra_ops += ', "r"(srcl)'
    return (f"// {what}: 4x4 outputs per lane, {WY}x{WX} input window\n"
            f"#define {name}(nch, desc_addr, vals_addr, win_addr, pitch_b, plane_b, tbase, edge{extra_args}) \\\n"
            f'    asm volatile("{body}" :: "r"(nch), "r"(desc_addr), "r"(vals_addr), "r"(win_addr), '
            f'"r"(pitch_b), "r"(plane_b), "r"(tbase), "r"(edge){extra_ops} : "memory")\n')


def generate() -> str:
    """The text of pattern_dispatch.h."""
    text = ["// generated by gen_dispatch.py -- do not edit", "#pragma once", ""]
    for S in STRIDES:
        for half in (False, True):
            text.append(macro(S, half))
            if S == 2:
                text.append(macro(S, half, groups=2))
                if not half:
                    text.append(macro(S, half, groups=2, dealt=True))
            if S == 1:
                text.append(macro(S, half, shift=1))
                if not half:
                    text.append(macro(S, half, shift=2))
    return "\n".join(text)


def main():
    with open(sys.argv[1], "w") as f:
        f.write(generate())


if __name__ == "__main__":
    main()
