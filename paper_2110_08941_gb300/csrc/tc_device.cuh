// Device-side building blocks shared by the tensor-core GEMM kernels (one-SM and SM-pair forms):
// PTX wrappers for mbarriers, TMA, tcgen05, the descriptors, tile decoding and the fused
// epilogue unit.  Internal to libhs.
#pragma once

#include "gemm_tc.cuh"

namespace hs {
namespace tcdev {

constexpr int BK = kTcBK;
constexpr int MN_CHUNK = 64 * BK * 2;                // one 64-wide MN slab of an MN-major tile (8 KB)
constexpr uint64_t kWaitLimitNs = 2000000000ull;     // 2 s per wait

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase with the given parity; false if the abort flag rises or the limit passes.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tm, int c0, int c1,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* tm, const int (&c)[4], uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], "
      "[%6];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tm)), "r"(c[0]), "r"(c[1]), "r"(c[2]), "r"(c[3]), "r"(bar)
      : "memory");
}
// Coordinates (channel, input column, input row, image) of the 4-D box holding implicit patch rows
// row..row+63 (row a multiple of 64) and patch columns kcol..kcol+63 (kcol a multiple of 64 below
// 9 * C): tap = kcol / C, channels kcol % C onwards, input pixel (stride * ho + kh - 1, kw - 1) for
// the block's first output pixel (ho, 0).
__device__ __forceinline__ void conv_box_coords(const TcConvGeom& g, int row, int kcol, int (&c)[4]) {
  const int blk = kcol >> 6;
  const int tap = blk / g.cblocks;
  const int cb = blk - tap * g.cblocks;
  const int img = row / g.hw;
  const int ho = (row - img * g.hw) / g.Wo;
  c[0] = cb * 64;
  c[1] = tap % 3 - 1;
  c[2] = g.stride * ho + tap / 3 - 1;
  c[3] = img;
}
// The same for the sub-pixel input gradient of class `cls` = 2 * ph + pw: patch column block
// kcol / 64 = (tap t of the class, Cout block); the class's row taps are kh = 1 (ph = 0) or kh = 0
// then 2 (ph = 1), which read output row a + 1 and a (dh = 1, 0); columns likewise.
__device__ __forceinline__ void subpixel_box_coords(const TcConvGeom& g, int cls, int row, int kcol,
                                                    int (&c)[4]) {
  const int blk = kcol >> 6;
  const int t = blk / g.cblocks;
  const int cb = blk - t * g.cblocks;
  const int ph = cls >> 1, pw = cls & 1;
  const int nw = pw ? 2 : 1;
  const int th = t / nw, tw = t - th * nw;
  const int img = row / g.hw;
  const int a = (row - img * g.hw) / g.Wo;
  c[0] = cb * 64;
  c[1] = (pw && tw == 0) ? 1 : 0;
  c[2] = a + ((ph && th == 0) ? 1 : 0);
  c[3] = img;
}
// The same coordinates in two parts, so a producer forms each part once per tile or per k-block
// instead of per box: the output-pixel part (image, first input row = stride * output row; for the
// sub-pixel product the class-grid row) and the patch-column part (channel block, column and row
// offsets of the tap).  Box coordinates: {c0, dw, h + dh, img}.
struct ConvRowPart { int img, h; };
struct ConvColPart { int c0, dw, dh; };
__device__ __forceinline__ ConvRowPart conv_row_part(const TcConvGeom& g, int row) {
  const int img = row / g.hw;
  const int ho = (row - img * g.hw) / g.Wo;
  return {img, g.stride * ho};
}
__device__ __forceinline__ ConvColPart conv_col_part(const TcConvGeom& g, int kcol) {
  const int blk = kcol >> 6;
  const int tap = blk / g.cblocks;
  const int cb = blk - tap * g.cblocks;
  return {cb * 64, tap % 3 - 1, tap / 3 - 1};
}
__device__ __forceinline__ ConvRowPart subpixel_row_part(const TcConvGeom& g, int row) {
  const int img = row / g.hw;
  return {img, (row - img * g.hw) / g.Wo};
}
__device__ __forceinline__ ConvColPart subpixel_col_part(const TcConvGeom& g, int cls, int kcol) {
  const int blk = kcol >> 6;
  const int t = blk / g.cblocks;
  const int cb = blk - t * g.cblocks;
  const int ph = cls >> 1, pw = cls & 1;
  const int nw = pw ? 2 : 1;
  const int th = t / nw, tw = t - th * nw;
  return {cb * 64, (pw && tw == 0) ? 1 : 0, (ph && th == 0) ? 1 : 0};
}
// The producers walk a tile's k-blocks in order, so instead of dividing per k-block (a long
// dependent chain on the single issuing thread, slower than the k-block's MMAs) they step these
// iterators: set up once per tile with divisions, then advanced by adds and compares.
// Patch-column blocks of the A operand (K-major): forward (sub < 0) block = tap * cblocks + cb with
// tap = 3 * kh + kw; sub-pixel class `sub` block = (th * nw + tw) * cblocks + cb.
struct ConvColIter {
  int cb, cblocks, a, na, b;   // forward: a = kw, b = kh (na = 3); sub-pixel: a = tw, b = th (na = nw)
  int ph, pw;                  // sub-pixel class parities; -1 for the forward
  __device__ __forceinline__ void init(const TcConvGeom& g, int sub, int kcol) {
    const int blk = kcol >> 6;
    cblocks = g.cblocks;
    const int t = blk / cblocks;
    cb = blk - t * cblocks;
    if (sub < 0) {
      ph = pw = -1;
      na = 3;
      b = t / 3;
      a = t - 3 * b;
    } else {
      ph = sub >> 1;
      pw = sub & 1;
      na = pw ? 2 : 1;
      b = t / na;
      a = t - b * na;
    }
  }
  __device__ __forceinline__ ConvColPart part() const {
    if (ph < 0) return {cb * 64, a - 1, b - 1};
    return {cb * 64, (pw && a == 0) ? 1 : 0, (ph && b == 0) ? 1 : 0};
  }
  __device__ __forceinline__ void next() {
    if (++cb == cblocks) {
      cb = 0;
      if (++a == na) {
        a = 0;
        ++b;
      }
    }
  }
};
// Output-pixel blocks of 64 rows of the implicit patch rows as the B operand (MN-major, K = pixels):
// 64 / Wo output rows per block within an image, or 64 / hw whole images per block.
struct ConvRowIter {
  int img, ho, Ho, dho, dimg, stride;
  __device__ __forceinline__ void init(const TcConvGeom& g, int row) {
    img = row / g.hw;
    ho = (row - img * g.hw) / g.Wo;
    Ho = g.hw / g.Wo;
    stride = g.stride;
    if (g.hw >= 64) {
      dho = 64 / g.Wo;
      dimg = 0;
    } else {
      dho = 0;
      dimg = 64 / g.hw;
    }
  }
  __device__ __forceinline__ ConvRowPart part() const { return {img, stride * ho}; }
  __device__ __forceinline__ void next() {
    if (dimg) {
      img += dimg;
    } else if ((ho += dho) >= Ho) {
      ho = 0;
      ++img;
    }
  }
};
__device__ __forceinline__ void conv_coords(const ConvRowPart& r, const ConvColPart& k, int (&c)[4]) {
  c[0] = k.c0;
  c[1] = k.dw;
  c[2] = r.h + k.dh;
  c[3] = r.img;
}

__device__ __forceinline__ void tma_store_4d(const CUtensorMap* tm, uint32_t src, const int (&c)[4]) {
  asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%1, %2, %3, %4}], [%5];"
               ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c[0]), "r"(c[1]), "r"(c[2]), "r"(c[3]), "r"(src)
               : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* tm, uint32_t src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
               ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(src)
               : "memory");
}
// Store the 32-row strip at rows row0.. (row0 a multiple of 32), columns n_base.. through the
// output map of the group: a 2-D [rows][cols] map, or (conv_d) a class grid of the input gradient.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* tm, uint32_t src, int c0, int c1, int c2) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];"
               ::"l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(src)
               : "memory");
}
template <bool CONV>
__device__ __forceinline__ void store_strip(const TcGemmParams& p, const CUtensorMap* td, uint32_t buf, int n_base,
                                            int row0, int part) {
  if (p.ksplit > 1) {
    tma_store_3d(td, buf, n_base, row0, part);
  } else if (CONV && p.conv_d) {
    const int img = row0 / p.conv.hw;
    int col = n_base;
    if (p.conv_d == 2) {   // column block = class: its own pixel grid
      const int cls = n_base / p.conv.cin_d;
      td = &p.tmD[cls];
      col = n_base - cls * p.conv.cin_d;
    }
    const int c[4] = {col, 0, (row0 - img * p.conv.hw) / p.conv.Wo, img};
    tma_store_4d(td, buf, c);
  } else {
    tma_store_2d(td, buf, n_base, row0);
  }
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// At most one bulk group may still be reading shared memory.
__device__ __forceinline__ void bulk_wait_read_1() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
// Programmatic dependent launch.  The GEMM kernels are launched with programmatic stream
// serialisation, so they may start while the previous kernel of the stream is finishing: each
// waits here, after its prologue (barriers, tensor memory, cluster sync) and before its first
// global-memory access, until that kernel has completed and its writes are visible; then it lets
// the next kernel of the stream start its own prologue on SMs as they free up.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dependents_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* tm) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
// 32 lanes x 32 consecutive fp32 columns: thread t receives row (quadrant base + t).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
// The wait names the destination registers so no use of them is scheduled above it.
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                 "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                 "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]),
                 "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]),
                 "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}

// Instruction descriptor, kind::f16: D fp32, A/B bf16, per-operand major-ness, N = BN, M = BM.
__host__ __device__ constexpr uint32_t make_idesc(bool a_mn, bool b_mn, int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

// Shared-memory matrix descriptor, 128-byte swizzle.  lbo/sbo in bytes.
//   K-major tile (rows x 64 K, 128 B per row, 8-row swizzle atoms of 1 KB): SBO = 1 KB between
//     8-row groups; LBO unused.  The K step of 16 elements advances the start by 32 B.
//   MN-major tile (64 K rows x 128 B per 64-wide MN slab): SBO = 1 KB between 8-row K groups,
//     LBO = 8 KB between 64-wide MN slabs.  The K step of 16 rows advances the start by 2 KB.
__device__ __forceinline__ uint64_t make_sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= 2ull << 61;
  return d;
}

__device__ __forceinline__ void record_error(DevStatus* st, int32_t code, int32_t info) {
  if (!st) return;
  if (st && atomicCAS(&st->err, 0, code) == 0) st->err_info = info;
}

struct TileCoord {
  int g, tm, tn;
};

// Tiles are numbered group-major; within a group, bands of 16 M-tiles are walked N-tile by
// N-tile so that the CTAs running at the same time share A and B panels in L2.
__device__ __forceinline__ TileCoord decode_tile(int t, int tiles_m, int tiles_n) {
  const int per_group = tiles_m * tiles_n;
  TileCoord c;
  c.g = t / per_group;
  const int r = t - c.g * per_group;
  constexpr int GM = 16;
  const int band = r / (GM * tiles_n);
  const int within = r - band * GM * tiles_n;
  const int rows = min(GM, tiles_m - band * GM);
  c.tm = band * GM + within % rows;
  c.tn = within / rows;
  return c;
}

// A tile's work: its coordinates, its group and split-K part, and its k-block range.  decode_tile's
// group index runs over groups x ksplit "virtual groups".
struct TileWork {
  TileCoord c;
  int g, part, kb_lo, kb_hi;
};
__device__ __forceinline__ int ksplit_of(const TcGemmParams& p) { return p.ksplit > 1 ? p.ksplit : 1; }
__device__ __forceinline__ TileWork tile_work(const TcGemmParams& p, int t, int tiles_m, int tiles_n) {
  TileWork w;
  w.c = decode_tile(t, tiles_m, tiles_n);
  if (p.ksplit > 1) {
    const int ks = p.ksplit;
    w.g = w.c.g / ks;
    w.part = w.c.g - w.g * ks;
    const int nkb = p.num_kb[w.g];
    w.kb_lo = nkb * w.part / ks;   // nkb * ks stays far below 2^31 (k-blocks of 64 rows, ks <= 304)
    w.kb_hi = nkb * (w.part + 1) / ks;
  } else {
    w.g = w.c.g;
    w.part = 0;
    w.kb_lo = 0;
    w.kb_hi = p.num_kb[w.g];
  }
  return w;
}

// MMA steps of 16 rows in group g's last k-block, whose rows past the group's extent are zero
// fill (their products add nothing): kb_last = that k-block (-1: issue all 4 everywhere).  Read
// once per group, outside the k-block loop: the issuing thread is on the tensor core's critical
// path, and a parameter load per k-block shows up in the main loop.
struct LastKb {
  int kb_last, steps;
};
__device__ __forceinline__ LastKb last_kb_of(const TcGemmParams& p, int g) {
  const int l = p.last_ksteps[g];
  LastKb r;
  r.kb_last = l > 0 ? p.num_kb[g] - 1 : -1;
  r.steps = l;
  return r;
}

// The one-SM MMAs of one k-block (four 16-row steps; see mma_kblock_pair), or of its first
// `steps` steps.
template <bool A_MN, bool B_MN>
__device__ __forceinline__ void mma_ksteps(uint32_t d_tmem, uint64_t ad, uint64_t bd, uint32_t idesc, uint32_t acc0,
                                           int steps) {
  constexpr uint64_t kA = A_MN ? (2048 >> 4) : (32 >> 4);
  constexpr uint64_t kB = B_MN ? (2048 >> 4) : (32 >> 4);
  if (steps == BK / 16) {
    umma_bf16(d_tmem, ad, bd, idesc, acc0);
    umma_bf16(d_tmem, ad + kA, bd + kB, idesc, 1u);
    umma_bf16(d_tmem, ad + 2 * kA, bd + 2 * kB, idesc, 1u);
    umma_bf16(d_tmem, ad + 3 * kA, bd + 3 * kB, idesc, 1u);
  } else {
#pragma unroll 1
    for (int kk = 0; kk < steps; ++kk) umma_bf16(d_tmem, ad + kk * kA, bd + kk * kB, idesc, kk ? 1u : acc0);
  }
}

__device__ __forceinline__ float u2f(uint32_t u) { return __uint_as_float(u); }

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&v);
}

// One epilogue unit: a 128-byte column strip of one accumulator row (32 fp32 or 64 bf16 outputs),
// computed from `r` (columns n_base..n_base+31) and, for bf16 outputs, `r2` (n_base+32..+63), packed
// into eight 16-byte words.  Columns past n_store are computed but never stored (the TMA store
// clips them); only the bias and mask reads are guarded.
// The mask operand of one kTcEpiMaskBf16 unit: Z's 64 bf16 values at (row, n_base..n_base+63) (for
// the sub-pixel input gradient, row is class pixel (a, b) of group grp = input pixel
// (2a + ph, 2b + pw)); zero past Mdim rows or n_store columns.  Loaded ahead of the accumulator
// so that the global-load latency overlaps the main loop.
template <bool CONV>
__device__ __forceinline__ void load_mask_unit(const TcGemmParams& p, int grp, int row, int n_base, uint4 (&zq)[8]) {
#pragma unroll
  for (int j = 0; j < 8; ++j) zq[j] = make_uint4(0u, 0u, 0u, 0u);
  if (row >= p.Mdim || n_base >= p.n_store) return;
  int64_t zrow = row;
  int col = n_base;
  if (CONV && p.conv_d) {
    if (p.conv_d == 2) {   // column block = class
      grp = n_base / p.conv.cin_d;
      col = n_base - grp * p.conv.cin_d;
    }
    const int img = row / p.conv.hw;
    const int rem = row - img * p.conv.hw;
    const int a = rem / p.conv.Wo, b = rem - a * p.conv.Wo;
    zrow = ((int64_t)img * p.conv.H + 2 * a + (grp >> 1)) * p.conv.W + 2 * b + (grp & 1);
  }
  if (p.relu_bits_in) {
    // the packed form of the same decisions, one 64-bit word per row of Z and 64-column unit
    const unsigned long long b =
        __ldg(reinterpret_cast<const unsigned long long*>(p.relu_bits_in) + (int64_t)(col >> 6) * p.bits_ld + zrow);
    zq[0].x = (uint32_t)b;
    zq[0].y = (uint32_t)(b >> 32);
    return;
  }
  const __nv_bfloat16* z = p.Z + zrow * p.ldz + col;
  if (n_base + 64 <= p.n_store) {
    const uint4* z4 = reinterpret_cast<const uint4*>(z);
#pragma unroll
    for (int j = 0; j < 8; ++j) zq[j] = __ldg(z4 + j);
  } else {
    uint16_t* zs = reinterpret_cast<uint16_t*>(zq);
    for (int j = 0; j < 64 && n_base + j < p.n_store; ++j) zs[j] = reinterpret_cast<const uint16_t*>(z)[j];
  }
}

template <int EPI, bool CONV>
__device__ __forceinline__ void epilogue_unit(const TcGemmParams& p, int grp, int row, int n_base,
                                              const uint32_t (&r)[32], const uint32_t (&r2)[32], const uint4 (&zq)[8],
                                              uint4 (&o)[8]) {
  if (EPI == kTcEpiStoreF32) {
#pragma unroll
    for (int j = 0; j < 8; ++j) o[j] = make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
  } else if (EPI == kTcEpiBiasF32) {
    float b[32];
    if (n_base + 32 <= p.Ndim) {
      const float4* b4 = reinterpret_cast<const float4*>(p.bias + n_base);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float4 t = __ldg(b4 + j);
        b[4 * j] = t.x; b[4 * j + 1] = t.y; b[4 * j + 2] = t.z; b[4 * j + 3] = t.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) b[j] = (n_base + j < p.Ndim) ? __ldg(p.bias + n_base + j) : 0.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      o[j] = make_uint4(__float_as_uint(u2f(r[4 * j]) + b[4 * j]), __float_as_uint(u2f(r[4 * j + 1]) + b[4 * j + 1]),
                        __float_as_uint(u2f(r[4 * j + 2]) + b[4 * j + 2]),
                        __float_as_uint(u2f(r[4 * j + 3]) + b[4 * j + 3]));
  } else {
    // bf16 outputs: 64 columns
    float v[64];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      v[j] = u2f(r[j]);
      v[32 + j] = u2f(r2[j]);
    }
    if (EPI == kTcEpiBiasReluBf16) {
      if (n_base + 64 <= p.Ndim) {
        const float4* b4 = reinterpret_cast<const float4*>(p.bias + n_base);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float4 t = __ldg(b4 + j);
          v[4 * j] = fmaxf(v[4 * j] + t.x, 0.f);
          v[4 * j + 1] = fmaxf(v[4 * j + 1] + t.y, 0.f);
          v[4 * j + 2] = fmaxf(v[4 * j + 2] + t.z, 0.f);
          v[4 * j + 3] = fmaxf(v[4 * j + 3] + t.w, 0.f);
        }
      } else {
#pragma unroll
        for (int j = 0; j < 64; ++j)
          v[j] = fmaxf(v[j] + ((n_base + j < p.Ndim) ? __ldg(p.bias + n_base + j) : 0.f), 0.f);
      }
    } else if (p.relu_bits_in) {   // kTcEpiMaskBf16, ReLU' from the packed bits (in zq[0])
      const uint64_t bits = (uint64_t)zq[0].x | ((uint64_t)zq[0].y << 32);
#pragma unroll
      for (int k = 0; k < 64; ++k) v[k] = ((bits >> k) & 1ull) ? v[k] : 0.f;
    } else {   // kTcEpiMaskBf16: ReLU' from the stored activation of the same row (prefetched in zq)
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t w[4] = {zq[j].x, zq[j].y, zq[j].z, zq[j].w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const __nv_bfloat162 pr = *reinterpret_cast<const __nv_bfloat162*>(&w[h]);
          const int k = 8 * j + 2 * h;
          v[k] = (__low2float(pr) > 0.f) ? v[k] : 0.f;
          v[k + 1] = (__high2float(pr) > 0.f) ? v[k + 1] : 0.f;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      o[j] = make_uint4(pack_bf16(v[8 * j], v[8 * j + 1]), pack_bf16(v[8 * j + 2], v[8 * j + 3]),
                        pack_bf16(v[8 * j + 4], v[8 * j + 5]), pack_bf16(v[8 * j + 6], v[8 * j + 7]));
    if (EPI == kTcEpiBiasReluBf16 && p.relu_bits_out && row < p.Mdim && n_base < p.n_store) {
      // ReLU' of the stored (bf16) activations for the input-gradient product: bit k = value > 0
      uint64_t bits = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t w[4] = {o[j].x, o[j].y, o[j].z, o[j].w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const __nv_bfloat162 pr = *reinterpret_cast<const __nv_bfloat162*>(&w[h]);
          const int k = 8 * j + 2 * h;
          bits |= (uint64_t)(__low2float(pr) > 0.f) << k;
          bits |= (uint64_t)(__high2float(pr) > 0.f) << (k + 1);
        }
      }
      reinterpret_cast<unsigned long long*>(p.relu_bits_out)[(int64_t)(n_base >> 6) * p.bits_ld + row] = bits;
    }
  }
}

}  // namespace tcdev
}  // namespace hs
