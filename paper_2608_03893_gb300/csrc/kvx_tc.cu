// Tensor-core mapping kernel for sm_103a (tcgen05 + TMEM + TMA), bf16 caches, bf16 or
// fp32 weights, head_dim 128, per-head features, half-split or interleaved RoPE pairs, k <= 4.
//
// It computes Eq. ridge_kv with the Sec. 3.3 RoPE composition,
//   K_t^{l,h} = R_t(t) ( [R_s(t)^-1 K_s^{sel[l][j]}[h]]_j W_K^{l,h} + b_K^{l,h} ),
//   V_t^{l,h} =          [V_s^{sel[l][j]}[h]]_j W_V^{l,h} + b_V^{l,h},
// with the stripped keys rounded to bf16 before the contraction and fp32 accumulation.
//
// The kernel runs as clusters of two CTAs (one per SM).  Work unit = (sequence b, pair of
// adjacent 128-token tiles, head h, K|V); CTA rank r of the cluster takes tile 2p + r.  A
// persistent cluster walks every target layer of a unit.  The k source tiles a target
// layer concatenates are the A operand of the contraction and live in tensor memory: four
// 64-column TMEM slots per CTA, each holding a 128-token x 128-feature bf16 tile (lane =
// token, two features per column).  A host-built schedule (Belady over the sequence of
// (layer, j) uses) keeps every source tile resident while later target layers still
// select it, so each source layer is read from HBM once per token tile and shared by all
// target layers that select it.  A slot is released as soon as the MMAs of its tile's
// last use complete, so the tile a layer adds is written while the rest of the previous
// layer still computes.
//
// Contraction of target layer l for both CTAs' tiles: D[256 tok x 128 ch] =
// X[256 x kd] W[kd x 128] as tcgen05 pair MMAs (cta_group::2, M = 256, N = 128, K = 16 per
// instruction), issued by the rank-0 CTA.  Each CTA supplies its 128 rows of A from its own
// TMEM and 64 of the 128 output channels of B = W^T from its own 16 KB shared-memory stage
// (64 rows x 128 features as two 64-feature halves, 128-byte swizzle); D lands in each
// CTA's own two 128-column fp32 TMEM accumulators.  Sharing B halves each SM's W traffic
// from L2 and the shared memory it needs per use, so each issuer's ring holds four uses.
// W needs no L2 prefetch: the clusters in flight share one (K|V, head) block.
//
// fp32 weights (the paper keeps W in fp32) are split on the host into bf16 hi = bf16(w)
// and lo = bf16(w - hi); each use then takes two W stages, hi and lo, whose MMAs read the
// same source tile and accumulate into the same TMEM accumulator, so X W = X W_hi + X W_lo
// to within 2^-17 of each weight.
//
// Cross-CTA hand-offs: both CTAs' W loads complete on the rank-0 CTA's stage barrier;
// both CTAs' prologue and epilogue warps arrive on the rank-0 CTA's tready / acce
// barriers; the rank-0 issuers' commits arrive on the wempty / tfree / accf barriers of
// both CTAs (multicast).
//
// Warp roles (512 threads; per-warpgroup register shares set with setmaxnreg):
//   warp 0      one thread polling two streams without blocking: TMA loads of raw source
//               tiles into the two landing buffers, and each layer's bias row
//   warp 1      TMEM allocator (all 512 columns, jointly with the peer CTA); in the rank-0
//               CTA, issuer of the even target layers
//   warp 3      in the rank-0 CTA, issuer of the odd target layers.  Each issuer owns one
//               accumulator, one ring of W stages and one tready/tfree barrier per slot.
//   warp 2      one thread polling the two W rings without blocking, one per issuer.  A
//               poll of shared memory costs hundreds of cycles under this kernel's
//               traffic, so each poller serves few streams.
//   warps 4-11  epilogue, two warpgroups (one warp per TMEM lane quarter, warp % 4).
//               Thread (group g, row r) owns token row r (= TMEM lane r) and the 32 RoPE
//               pairs 32g .. 32g+31 (channels i and i + 64): TMEM -> registers, + bias,
//               (keys) target RoPE, bf16.  Every layer loads both halves of its
//               accumulator at once and releases it before any arithmetic; the register
//               split (32 / 160 / 160) gives the epilogue room for the 64 accumulator words
//               beside a key unit's cos / sin of 32 pairs.  Key and value units run
//               separate instances of the layer loop (values carry no cos / sin).
//               For a contiguous target each warp stages its
//               32 rows x 2 x 32 channels (64-byte swizzle) and writes them with its own
//               TMA stores; a warp with a row at an out-of-range position writes its valid
//               rows directly.  Paged targets take 16-byte stores through the block table.
//   warps 12-15 prologue, one warpgroup (one warp per lane quarter); thread r owns token
//               row r and all 64 pairs: landing buffer -> registers -> (keys) strip the
//               source RoPE in fp32, round to bf16 -> tcgen05.st into the tile's TMEM slot.
//               Running the prologue on its own warps takes it off the epilogue's per-layer
//               chain of waits, loads and stores.
//
// Every mbarrier wait is bounded: after 4 s the kernel raises KVX_ERR_TIMEOUT in the
// status word, sets a shared abort flag that every role polls, waits (again bounded)
// for its own TMA copies and MMAs in flight, frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>
#include <type_traits>
#include <vector>

#include "kvx_internal.h"
#include "kvx_ptx.cuh"
#include "kvx_rope.cuh"
#include "kvx_xh.h"

namespace kvx {
namespace {

using namespace ptx;

constexpr int kThreads = 512;
constexpr int kFirstEpiWarp = 4;                    // warps 4-11: epilogue
constexpr int kEpiWarps = 8;
constexpr int kFirstProWarp = 12;                   // warps 12-15: prologue
constexpr int kProWarps = 4;
// Registers per thread of each warpgroup (setmaxnreg): the control warps give up most of
// theirs so that the epilogue keeps its cos/sin of 32 pairs beside a whole accumulator row
// (64 words) and the prologue its cos/sin of all 64 pairs in registers.  The shares add up
// to the launch's 128 x 512.
constexpr uint32_t kRegsCtl = 32, kRegsEpi = 160, kRegsPro = 160;
static_assert(kRegsCtl * 128 + kRegsEpi * 256 + kRegsPro * 128 <= 128u * kThreads,
              "register split exceeds the launch's register file share");
constexpr int kTileM = 128;                         // tokens per work unit
constexpr int kD = 128;                             // head_dim of this kernel
constexpr uint32_t kLandBytes = kTileM * kD * 2;    // 32 KB raw tile: two 64-column SW128 halves
constexpr uint32_t kHalfBytes = kLandBytes / 2;     // 16 KB
constexpr uint32_t kWStageBytes = (kD / 2) * 128 * 2; // 16 KB: this CTA's 64 output rows of one use
                                                      // (two 64-feature halves)
constexpr uint32_t kPieceBytes = 32 * 64;           // 2 KB: 32 rows x 32 channels, 64-byte swizzle
constexpr uint32_t kWarpStageBytes = 2 * kPieceBytes; // one epilogue warp's share of an output tile
constexpr int kStageBufs = 1;                       // staging buffers per epilogue warp
constexpr uint32_t kOutBytes = kStageBufs * kEpiWarps * kWarpStageBytes;
constexpr int kTSlots = 4;                          // TMEM source-tile slots (64 columns each)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCols = 128;                  // one fp32 accumulator
constexpr int kAccBufs = 2;
constexpr uint32_t kSlotCol0 = kAccBufs * kAccCols; // 256: first source-slot column
constexpr int kLand = 2;                            // landing buffers for raw source tiles
constexpr int kIssuers = 2;                         // MMA-issuing threads (even / odd target layers)
constexpr int kBiasSlots = 4;                       // per-layer bias rows staged ahead (512 B each)
constexpr uint32_t kBiasBytes = kD * 4;
constexpr size_t kSmemLimit = 232448;               // 227 KB opt-in per CTA

constexpr int kRing = 4;                            // W stages (uses) per issuer ring
constexpr int kNW = kRing * kIssuers;               // W stages in shared memory

// Dynamic shared memory: the 128-byte-swizzled buffers need 1024-byte alignment, which
// the base of the dynamic window has (the kernel checks it) since nothing else is placed
// before it; no slack is reserved.
constexpr size_t smem_bytes() {
  return static_cast<size_t>(kLand) * kLandBytes + static_cast<size_t>(kNW) * kWStageBytes +
         kOutBytes + kBiasSlots * kBiasBytes +
         (2 * kLand + 2 * kTSlots * kIssuers + 2 * kNW + 2 * kAccBufs + 2 * kBiasSlots + kIssuers) * 8 + 16;
}
static_assert(smem_bytes() <= kSmemLimit, "shared-memory layout exceeds the per-CTA limit");
static_assert(kRing >= 2, "each W ring must hold two uses");

struct TcParams {
  CUtensorMap tm_k;      // source keys   [L_s][B][H][T][128] bf16, box 64 x 128
  CUtensorMap tm_v;      // source values
  CUtensorMap tm_w;      // W^T [L_t*2*H*128][F] bf16 (fp32 weights: [hi | lo], 2F columns), box 64 x 64
  CUtensorMap tm_out_k;  // target keys as (64 ch, T, 2 halves, B*H or H, L_t), box 32 x 32 x 2 x 1 x 1
  CUtensorMap tm_out_v;  // target values (contiguous targets whose (batch, head) dims merge)
  MapArgs a;
  const int32_t* load_layer;   // [n_loads] source layer of load e
  const int32_t* load_slot;    // [n_loads] TMEM slot
  const uint32_t* use_pack;    // [L_t] per use j: 5 bits at 5j = slot | 4 first use | 16 release after
  const float* bias;           // [L_t][2][H][128] fp32
  int32_t* status;
  int32_t Lt, H, k, n_loads, tiles_per_seq, n_units;   // tiles_per_seq / n_units count pairs of token tiles
  int32_t out_bh;        // TMA-store head coordinate: 0 none (direct stores), 1 h (B = 1), 2 b*H + h
  RopeTables rope;
  uint64_t timeout_ns;   // bound of every wait (kTimeoutNs unless a test shortens it)
  int32_t skip_bias;     // test only: CTA 0 never loads its bias row of this index (-1: none)
};

struct Unit {
  int b, t0, h, kv;
};

// Units (tile pairs) are visited u = cluster + i * clusters, tile pair fastest, then
// sequence, head, and K|V outermost.  The clusters running at any moment then work on one
// or two (K|V, head) pairs, so the W^T rows they stream (8 MB per pair at L_t = 64, k = 4)
// stay in L2 even when the clusters drift to different target layers; every cluster still
// gets nearly equal numbers of (heavier) key and value units.  Rank 1's tile of the last
// pair lies past the sequence end when the tile count is odd: its rows are all masked.
__device__ __forceinline__ Unit decode_unit(int u, int H, int B, int pairs, uint32_t rank) {
  Unit r;
  r.t0 = (2 * (u % pairs) + static_cast<int>(rank)) * kTileM;   // past the end for an odd tile count
  int rest = u / pairs;
  r.b = rest % B;
  rest /= B;
  r.h = rest % H;
  r.kv = rest / H;
  return r;
}

__device__ __forceinline__ void report(int32_t* status, int code) { atomicCAS(status, 0, code); }

// Rotation of two RoPE pairs (x0.x, x1.x) and (x0.y, x1.y) by the angles with cosines c and
// sines s, one f32x2 instruction per step (each lane rounds like the scalar fmul / fma it
// replaces).  Strip (rotation by -t*omega): x0' = x0 c + x1 s, x1' = x1 c - x0 s; the sums
// are left unrounded for the bf16 pack.  Apply (rotation by +t*omega): y0' = y0 c - y1 s,
// y1' = y0 s + y1 c.  kHF: the operands are bf16 values, every product is rounded to bf16.
template <bool kHF>
__device__ __forceinline__ void rope_strip2(float2 x0, float2 x1, float2 c, float2 s, float2& r0, float2& r1) {
  if constexpr (kHF) {
    const float2 ac = bf16_round2(__fmul2_rn(x0, c)), bs = bf16_round2(__fmul2_rn(x1, s));
    const float2 bc = bf16_round2(__fmul2_rn(x1, c)), as = bf16_round2(__fmul2_rn(x0, s));
    r0 = make_float2(__fadd_rn(ac.x, bs.x), __fadd_rn(ac.y, bs.y));
    r1 = make_float2(__fsub_rn(bc.x, as.x), __fsub_rn(bc.y, as.y));
  } else {
    const float2 as = __fmul2_rn(x0, s);
    r0 = __ffma2_rn(x0, c, __fmul2_rn(x1, s));
    r1 = __ffma2_rn(x1, c, make_float2(-as.x, -as.y));
  }
}

// kHF: the mapped key is first rounded to bf16 (the tensor the forward rotates).
template <bool kHF>
__device__ __forceinline__ void rope_apply2(float2 y0, float2 y1, float2 c, float2 s, float2& r0, float2& r1) {
  if constexpr (kHF) {
    const float2 b0 = bf16_round2(y0), b1 = bf16_round2(y1);
    const float2 p0 = bf16_round2(__fmul2_rn(b0, c)), p1 = bf16_round2(__fmul2_rn(b1, s));
    const float2 p2 = bf16_round2(__fmul2_rn(b1, c)), p3 = bf16_round2(__fmul2_rn(b0, s));
    r0 = make_float2(__fsub_rn(p0.x, p1.x), __fsub_rn(p0.y, p1.y));
    r1 = make_float2(__fadd_rn(p2.x, p3.x), __fadd_rn(p2.y, p3.y));
  } else {
    const float2 u = __fmul2_rn(y1, s);
    r0 = __ffma2_rn(y0, c, make_float2(-u.x, -u.y));
    r1 = __ffma2_rn(y0, s, __fmul2_rn(y1, c));
  }
}

// ------------------------------------------------------------------------ kernel --

// kHF: the Hugging Face forward's RoPE rounding (kvx_rope_numerics): cos / sin of the fp32
// angle rounded to bf16, every product and sum of the rotations rounded to bf16.
// kParts: W stages per use, 1 for bf16 weights, 2 (hi, lo) for fp32 weights.
// kIL: interleaved RoPE pairs (2i, 2i+1) instead of half-split pairs (i, i + 64).
template <bool kHF, int kParts, bool kIL>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    tc_map_kernel(const __grid_constant__ TcParams P) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_u32(smem) & 1023u) {   // uniform over the CTA: every thread returns here
    if (threadIdx.x == 0) report(P.status, KVX_ERR_UNSUPPORTED);
    return;
  }
  uint8_t* land = smem;
  uint8_t* wst = land + kLand * kLandBytes;            // [2 rings][kRing] W stages
  uint8_t* outst = wst + static_cast<size_t>(kNW) * kWStageBytes;
  float* bias_ring = reinterpret_cast<float*>(outst + kOutBytes);   // [4][128] fp32
  uint64_t* bars = reinterpret_cast<uint64_t*>(bias_ring + kBiasSlots * kD);
  uint64_t* land_full = bars;                    // [2] TMA landed
  uint64_t* land_empty = land_full + kLand;      // [2] prologue read it (4 warps)
  uint64_t* tready = land_empty + kLand;         // [4][2] TMEM tile written for issuer i (4 warps x 2 CTAs)
  uint64_t* tfree = tready + kTSlots * kIssuers; // [4][2] TMEM tile released by issuer i
  uint64_t* wfull = tfree + kTSlots * kIssuers;  // [2][kRing]
  uint64_t* wempty = wfull + kNW;                // [2][kRing]
  uint64_t* accf = wempty + kNW;                 // [2] accumulator ready
  uint64_t* acce = accf + kAccBufs;              // [2] accumulator drained (8 warps x 2 CTAs)
  uint64_t* bias_full = acce + kAccBufs;         // [4] bias row landed
  uint64_t* bias_empty = bias_full + kBiasSlots; // [4] bias row used (8 warps)
  uint64_t* drain = bias_empty + kBiasSlots;     // [2] per issuer
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + kIssuers);
  volatile uint32_t* abort_flag = tmem_holder + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();        // 0: issues the pair's MMAs
  const int unit0 = blockIdx.x >> 1, unit_step = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kLand; ++i) {
      mbar_init(smem_u32(&land_full[i]), 1);
      mbar_init(smem_u32(&land_empty[i]), kProWarps);
    }
    for (int i = 0; i < kTSlots * kIssuers; ++i) mbar_init(smem_u32(&tready[i]), 2 * kProWarps);
    for (int i = 0; i < kTSlots * kIssuers; ++i) mbar_init(smem_u32(&tfree[i]), 1);
    for (int i = 0; i < kNW; ++i) {
      mbar_init(smem_u32(&wfull[i]), 1);
      mbar_init(smem_u32(&wempty[i]), 1);
    }
    for (int i = 0; i < kAccBufs; ++i) {
      mbar_init(smem_u32(&accf[i]), 1);
      mbar_init(smem_u32(&acce[i]), 2 * kEpiWarps);
    }
    for (int i = 0; i < kBiasSlots; ++i) {
      mbar_init(smem_u32(&bias_full[i]), 1);
      mbar_init(smem_u32(&bias_empty[i]), kEpiWarps);
    }
    for (int i = 0; i < kIssuers; ++i) mbar_init(smem_u32(&drain[i]), 1);
    *abort_flag = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    // one warp of each CTA of the pair allocates, collectively, the same columns in both
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();   // the peer's barriers are initialised before any arrival from this CTA
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int Lt = P.Lt, k = P.k, H = P.H;
  const int n_units = P.n_units, tiles = P.tiles_per_seq;
  const MapArgs& A = P.a;
  // Each warpgroup takes its register share (every warp of it executes the same
  // setmaxnreg) before its warps go their separate ways.
  if (warp < kFirstEpiWarp) {
  setmaxnreg_dec<kRegsCtl>();
  if (warp == 0) {
    // ------------------------------------------- source-tile and bias producer ------
    // One thread polls two streams without blocking: the source tiles of the schedule
    // into the landing buffers, and every layer's bias row into the bias ring.  There is
    // no L2 prefetch of upcoming source tiles: under this kernel's streaming traffic a
    // tile prefetched a few loads ahead was often evicted before its load.
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t gl = 0, bn = 0;
      int su = unit0, se = 0, bu = unit0, blay = 0;
      Unit sun = decode_unit(su < n_units ? su : 0, H, A.B, tiles, rank);
      Unit bun = sun;
      bool ok = true;
      uint64_t t_idle = 0;
      uint32_t spins = 0;
      // a test's planted fault: this bias row is never loaded, so the epilogue's wait for
      // it runs out and the whole kernel takes its abort path
      const int64_t skip = blockIdx.x == 0 ? P.skip_bias : -1;
      for (;;) {
        bool busy = false, progress = false;
        if (su < n_units && P.n_loads > 0) {
          busy = true;
          const int lb = static_cast<int>(gl % kLand);
          const uint32_t round = gl / kLand;
          if (round == 0 || mbar_test_wait(smem_u32(&land_empty[lb]), (round - 1) & 1u)) {
            const int L = __ldg(&P.load_layer[se]);
            const CUtensorMap* tm = sun.kv ? &P.tm_v : &P.tm_k;
            const uint32_t dst = smem_u32(land + static_cast<size_t>(lb) * kLandBytes);
            mbar_expect_tx(smem_u32(&land_full[lb]), kLandBytes);
            tma_load_5d(dst, tm, smem_u32(&land_full[lb]), 0, sun.t0, sun.h, sun.b, L, pol);
            tma_load_5d(dst + kHalfBytes, tm, smem_u32(&land_full[lb]), 64, sun.t0, sun.h, sun.b, L, pol);
            ++gl;
            if (++se == P.n_loads) {
              se = 0;
              su += unit_step;
              if (su < n_units) sun = decode_unit(su, H, A.B, tiles, rank);
            }
            progress = true;
          }
        }
        if (bu < n_units) {
          busy = true;
          const int bs = static_cast<int>(bn % kBiasSlots);
          const uint32_t round = bn / kBiasSlots;
          if (round == 0 || mbar_test_wait(smem_u32(&bias_empty[bs]), (round - 1) & 1u)) {
            const int row0 = ((blay * 2 + bun.kv) * H + bun.h) * kD;
            if (static_cast<int64_t>(bn) != skip) {
              mbar_expect_tx(smem_u32(&bias_full[bs]), kBiasBytes);
              bulk_load(smem_u32(bias_ring + bs * kD), P.bias + static_cast<size_t>(row0), kBiasBytes,
                        smem_u32(&bias_full[bs]));
            }
            ++bn;
            if (++blay == Lt) {
              blay = 0;
              bu += unit_step;
              if (bu < n_units) bun = decode_unit(bu, H, A.B, tiles, rank);
            }
            progress = true;
          }
        }
        if (!busy) break;
        if (progress) {
          spins = 0;
          t_idle = 0;
          continue;
        }
        if ((++spins & 63u) == 0) {   // bounded: no slot freed for 4 s raises KVX_ERR_TIMEOUT
          if (*abort_flag) {
            ok = false;
            break;
          }
          const uint64_t now = global_timer();
          if (t_idle == 0) {
            t_idle = now;
          } else if (now - t_idle > P.timeout_ns) {
            *abort_flag = 1u;
            report(P.status, KVX_ERR_TIMEOUT);
            ok = false;
            break;
          }
        }
      }
      if (!ok) {   // the most recent loads and bias rows may still be landing
        const uint32_t first = gl > static_cast<uint32_t>(kLand) ? gl - kLand : 0;
        for (uint32_t i = first; i < gl; ++i)
          drain_wait(smem_u32(&land_full[i % kLand]), (i / kLand) & 1u, P.timeout_ns);
        const uint32_t bfirst = bn > static_cast<uint32_t>(kBiasSlots) ? bn - kBiasSlots : 0;
        for (uint32_t i = bfirst; i < bn; ++i)
          if (static_cast<int64_t>(i) != skip)
            drain_wait(smem_u32(&bias_full[i % kBiasSlots]), (i / kBiasSlots) & 1u, P.timeout_ns);
      }
    }
  } else if (warp == 2) {
    // ----------------------------------------------------------- W producer ------
    // One thread polls the W ring of each issuer (the k kParts stages of every layer of
    // its parity, in order) without blocking: a blocking wait on one ring would starve
    // the other issuer.
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();
      const int chunks = k * kParts;   // stages per layer: one 128-feature stage per use and part
      int wu[kIssuers], wl[kIssuers], wc[kIssuers], wkv[kIssuers], wh[kIssuers];
      uint32_t wn[kIssuers];     // stages filled into ring r
      for (int r = 0; r < kIssuers; ++r) {
        wu[r] = unit0;
        wl[r] = r;
        wc[r] = 0;
        wn[r] = 0;
        const Unit un = decode_unit(wu[r] < n_units ? wu[r] : 0, H, A.B, tiles, rank);
        wkv[r] = un.kv;
        wh[r] = un.h;
      }
      bool ok = true;
      uint64_t t_idle = 0;
      uint32_t spins = 0;
      for (;;) {
        bool busy = false, progress = false;
#pragma unroll
        for (int r = 0; r < kIssuers; ++r) {
          if (wl[r] >= Lt || wu[r] >= n_units) continue;   // done (or issuer r has no layer)
          busy = true;
          const int st = r * kRing + static_cast<int>(wn[r] % kRing);
          const uint32_t round = wn[r] / kRing;
          if (round > 0 && !mbar_test_wait(smem_u32(&wempty[st]), (round - 1) & 1u)) continue;
          // the layer (and unit) this ring fills after the current one
          int nl = wl[r] + kIssuers, nu = wu[r], nkv = wkv[r], nh = wh[r];
          if (nl >= Lt) {
            nl = r;
            nu += unit_step;
            if (nu < n_units) {
              const Unit nun = decode_unit(nu, H, A.B, tiles, rank);
              nkv = nun.kv;
              nh = nun.h;
            }
          }
          // this CTA's 64 of the use's 128 output rows; both CTAs' halves complete on the
          // rank-0 CTA's wfull, which expects the bytes of both
          if (rank == 0) mbar_expect_tx(smem_u32(&wfull[st]), 2 * kWStageBytes);
          const uint32_t wdst = smem_u32(wst + static_cast<size_t>(st) * kWStageBytes);
          const uint32_t wbar = mapa_shared(smem_u32(&wfull[st]), 0);
          const int wrow = ((wl[r] * 2 + wkv[r]) * H + wh[r]) * kD + static_cast<int>(rank) * (kD / 2);
          // stage c of a layer: use j = c / kParts, part p = c % kParts at W^T column p F + 128 j
          const int wx = (wc[r] % kParts) * k * 128 + (wc[r] / kParts) * 128;
          tma_load_2d_pair(wdst, &P.tm_w, wbar, wx, wrow, pol);
          tma_load_2d_pair(wdst + kWStageBytes / 2, &P.tm_w, wbar, wx + 64, wrow, pol);
          ++wn[r];
          if (++wc[r] == chunks) {
            wc[r] = 0;
            wl[r] = nl;
            wu[r] = nu;
            wkv[r] = nkv;
            wh[r] = nh;
          }
          progress = true;
        }
        if (!busy) break;
        if (progress) {
          spins = 0;
          t_idle = 0;
          continue;
        }
        if ((++spins & 63u) == 0) {   // bounded: no slot freed for 4 s raises KVX_ERR_TIMEOUT
          if (*abort_flag) {
            ok = false;
            break;
          }
          const uint64_t now = global_timer();
          if (t_idle == 0) {
            t_idle = now;
          } else if (now - t_idle > P.timeout_ns) {
            *abort_flag = 1u;
            report(P.status, KVX_ERR_TIMEOUT);
            ok = false;
            break;
          }
        }
      }
      if (!ok && rank == 0) {   // the most recent fills of each ring (both CTAs' halves) may still be landing
        for (int r = 0; r < kIssuers; ++r) {
          const uint32_t first = wn[r] > static_cast<uint32_t>(kRing) ? wn[r] - kRing : 0;
          for (uint32_t i = first; i < wn[r]; ++i)
            drain_wait(smem_u32(&wfull[r * kRing + i % kRing]), (i / kRing) & 1u, P.timeout_ns);
        }
      }
    }
  } else {   // warps 1 and 3
    // --------------------------------------------------------- MMA issuers --------
    // Warp 1 issues the even target layers into accumulator 0, warp 3 the odd ones into
    // accumulator 1.  A thread that reads shared memory (an mbarrier wait) while its own
    // MMAs are queued stalls for about as long as they take to start, so a single issuer
    // leaves the tensor pipe idle at every wait; with two issuers on different SM
    // sub-partitions the other one's queued MMAs cover it.
    const int iss = warp == 1 ? 0 : 1;
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = make_idesc(2 * kTileM, kD);   // M = 256: both CTAs' token tiles
      const uint32_t d_tmem = tmem_base + iss * kAccCols;
      uint32_t ready_par = 0, acc_n = 0, wi = 0;   // wi: W stages consumed from this issuer's ring
      bool ok = true, issued = false;
      uint32_t pack_next = iss < Lt ? __ldg(&P.use_pack[iss]) : 0u;
      for (int u = unit0; ok && u < n_units; u += unit_step) {
        for (int l = iss; ok && l < Lt; l += kIssuers, ++acc_n) {
          const uint32_t pack = pack_next;
          const int ln = l + kIssuers < Lt ? l + kIssuers : iss;
          pack_next = __ldg(&P.use_pack[ln]);   // schedule word of this issuer's next layer
          if (acc_n >= 1 && !wait_bar(smem_u32(&acce[iss]), (acc_n - 1) & 1u, abort_flag, P.status,
                                         KVX_ERR_TIMEOUT, P.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          for (int j = 0; ok && j < k; ++j) {
            // use bits: slot | 4 first use of the tile by this issuer | 16 release the
            // slot after this use.  The prologue warps signal tready[slot][issuer] only
            // for the loads this issuer uses, so it waits for every phase in order.
            const uint32_t f = (pack >> (5 * j)) & 31u;
            const uint32_t s = f & 3u;
            if (f & 4u) {
              if (!wait_bar(smem_u32(&tready[s * kIssuers + iss]), (ready_par >> s) & 1u, abort_flag,
                               P.status, KVX_ERR_TIMEOUT, P.timeout_ns)) {
                ok = false;
                break;
              }
              ready_par ^= 1u << s;
              tc_fence_after();   // the tile was written by other threads' tcgen05.st
            }
            const uint32_t a_col = tmem_base + kSlotCol0 + s * 64;
#pragma unroll
            for (int p = 0; p < kParts; ++p, ++wi) {   // hi (and lo) stages of this use
              const uint32_t st0 = iss * kRing + wi % kRing;
              if (!wait_bar(smem_u32(&wfull[st0]), (wi / kRing) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT,
                            P.timeout_ns)) {
                ok = false;
                break;
              }
              const uint32_t b0 = smem_u32(wst + static_cast<size_t>(st0) * kWStageBytes);
              const uint32_t b1 = b0 + kWStageBytes / 2;
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                tc_mma_ts_pair(d_tmem, a_col + kk * 8, sw128_desc(b0 + kk * 32), idesc, (j | p | kk) != 0);
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                tc_mma_ts_pair(d_tmem, a_col + 32 + kk * 8, sw128_desc(b1 + kk * 32), idesc, true);
              issued = true;
              tc_commit_pair(smem_u32(&wempty[st0]), 3);
            }
            if (ok && (f & 16u)) tc_commit_pair(smem_u32(&tfree[s * kIssuers + iss]), 3);
          }
          if (ok) tc_commit_pair(smem_u32(&accf[iss]), 3);
        }
      }
      // every MMA (and every commit) of this issuer must have completed before TMEM is freed
      if (issued || !ok) {
        tc_commit_pair(smem_u32(&drain[iss]), 1);
        drain_wait(smem_u32(&drain[iss]), 0, P.timeout_ns);
      }
    }
  }
  } else if (warp < kFirstProWarp) {
    setmaxnreg_inc<kRegsEpi>();
    // -------------------------------------------------------- epilogue warps ------
    const int g = (warp - kFirstEpiWarp) >> 2;       // pair group: pairs 32g .. 32g+31
    const int q = warp & 3;                          // TMEM lane quarter this warp may access
    const int r = q * 32 + lane;                     // token row within the tile
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    const uint64_t st_pol = policy_evict_first();
    uint32_t lay = 0, acc_n0 = 0, acc_n1 = 0;
    uint8_t* wstage = outst + static_cast<size_t>(warp - kFirstEpiWarp) * kStageBufs * kWarpStageBytes;
    float cs[32], sn[32];
    bool ok = true;
    for (int u = unit0; ok && u < n_units; u += unit_step) {
      const Unit un = decode_unit(u, H, A.B, tiles, rank);
      const int t = un.t0 + r;
      bool valid = t < A.T;
      bool bad = false;
      int p = 0;
      if (valid) {
        p = __ldg(&A.pos[static_cast<int64_t>(un.b) * A.T + t]);
        if (p < 0 || p >= (1 << 24)) {
          report(P.status, KVX_ERR_DEVICE_BOUNDS);
          valid = false;
          bad = true;
          p = 0;
        }
      }
      int64_t row_off = 0;
      if (valid) {
        if (!A.paged) {
          row_off = un.b * A.ts[1] + un.h * A.ts[2] + static_cast<int64_t>(t) * A.ts[3];
        } else {
          const int lb = p / A.block_size;
          const int blk =
              lb < A.max_blocks ? __ldg(&A.block_table[static_cast<int64_t>(un.b) * A.max_blocks + lb]) : -1;
          if (blk < 0 || blk >= A.n_blocks) {
            report(P.status, KVX_ERR_DEVICE_BOUNDS);
            valid = false;
          } else {
            row_off = static_cast<int64_t>(blk) * A.ts[1] + un.h * A.ts[2] +
                      static_cast<int64_t>(p % A.block_size) * A.ts[3];
          }
        }
      }
      // contiguous targets: each warp stages its 32 rows and writes them with TMA stores,
      // unless one of its rows has an out-of-range position: then its valid rows are
      // written directly (rows past the sequence end are clipped by the tensor map)
      const bool warp_tma = P.out_bh != 0 && __ballot_sync(0xffffffffu, bad) == 0u;
      if (un.kv == 0) {
#pragma unroll
        for (int m = 0; m < 32; ++m) {
          // pair of slot m: half-split pairs (c, c + 64) for c = 32g + m; interleaved pairs
          // (c, c + 1) for the 16 even c in [32g, 32g + 32) (m < 16), then in 64 + [32g, 32g + 32)
          const int i = kIL ? (m < 16 ? 16 * g + m : 32 + 16 * g + (m - 16)) : 32 * g + m;
          if constexpr (kHF) {
            sincosf(__fmul_rn(static_cast<float>(p), P.rope.wt_hi[i]), &sn[m], &cs[m]);
            sn[m] = bf16_round(sn[m]);
            cs[m] = bf16_round(cs[m]);
          } else {
            rope_sincos(p, P.rope.wt_hi[i], P.rope.wt_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi,
                        &sn[m], &cs[m]);
          }
        }
      }
      __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(un.kv ? A.tgt_v : A.tgt_k);
      const CUtensorMap* tm_out = un.kv ? &P.tm_out_v : &P.tm_out_k;
      // key and value units run separate instances of the layer loop (values carry no
      // cos / sin); each layer loads both halves of its accumulator at once and releases it
      // to the issuer before the arithmetic
      auto layers = [&](auto kv_tag) {
        constexpr bool kV = decltype(kv_tag)::value;
        for (int l = 0; ok && l < Lt; ++l, ++lay) {
          const uint32_t bslot = lay % kBiasSlots;
          const float* bias = bias_ring + bslot * kD;
          {
            const bool w_ok = wait_bar(smem_u32(&bias_full[bslot]), (lay / kBiasSlots) & 1u, abort_flag, P.status,
                                       KVX_ERR_TIMEOUT, P.timeout_ns);
            if (!__all_sync(0xffffffffu, w_ok)) {
              ok = false;
              break;
            }
          }
          const uint32_t buf = static_cast<uint32_t>(l) & 1u;   // accumulator of issuer l % 2
          {
            const uint32_t acc_par = (buf ? acc_n1 : acc_n0) & 1u;
            if (buf) ++acc_n1; else ++acc_n0;
            const bool w_ok = wait_bar(smem_u32(&accf[buf]), acc_par, abort_flag, P.status, KVX_ERR_TIMEOUT,
                                       P.timeout_ns);
            if (!__all_sync(0xffffffffu, w_ok)) {
              ok = false;
              break;
            }
          }
          tc_fence_after();
          // this warp's staging buffer for the layer; the store that last read it (this
          // thread's bulk group kStageBufs layers ago) must be done reading
          uint8_t* sb = wstage + (lay % kStageBufs) * kWarpStageBytes;
          if (!A.paged && lay >= static_cast<uint32_t>(kStageBufs)) {
            if (lane == 0) {
              if constexpr (kStageBufs == 1) bulk_wait_read_all(); else bulk_wait_read_but_last();
            }
            __syncwarp();
          }
          const uint32_t col = tmem_base + lane_addr + buf * kAccCols + 32 * g;
          auto release = [&] {   // the accumulator is free for the issuer's next layer
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&acce[buf]), 0));
          };
          uint32_t lo2[2][16], hi2[2][16];
          tmem_ld_2x16(col, col + 64, lo2[0], hi2[0]);
          tmem_ld_2x16(col + 16, col + 80, lo2[1], hi2[1]);
          release();
#pragma unroll
          for (int rnd = 0; rnd < 2; ++rnd) {
            uint32_t(&lo)[16] = lo2[rnd];
            uint32_t(&hi)[16] = hi2[rnd];
            const int c_lo = 32 * g + 16 * rnd;   // channels c_lo + [0,16) and 64 + c_lo + [0,16)
            float ylo[16], yhi[16];
#pragma unroll
            for (int j = 0; j < 16; j += 4) {
              const float4 b0 = *reinterpret_cast<const float4*>(bias + c_lo + j);
              const float4 b1 = *reinterpret_cast<const float4*>(bias + 64 + c_lo + j);
              ylo[j] = __fadd_rn(__uint_as_float(lo[j]), b0.x);
              ylo[j + 1] = __fadd_rn(__uint_as_float(lo[j + 1]), b0.y);
              ylo[j + 2] = __fadd_rn(__uint_as_float(lo[j + 2]), b0.z);
              ylo[j + 3] = __fadd_rn(__uint_as_float(lo[j + 3]), b0.w);
              yhi[j] = __fadd_rn(__uint_as_float(hi[j]), b1.x);
              yhi[j + 1] = __fadd_rn(__uint_as_float(hi[j + 1]), b1.y);
              yhi[j + 2] = __fadd_rn(__uint_as_float(hi[j + 2]), b1.z);
              yhi[j + 3] = __fadd_rn(__uint_as_float(hi[j + 3]), b1.w);
            }
            if (!kV && !kIL) {
              // target RoPE on pairs (c, c + 64): channel c_lo + j of ylo with the same of yhi
#pragma unroll
              for (int j = 0; j < 16; j += 2) {
                const float2 c = make_float2(cs[16 * rnd + j], cs[16 * rnd + j + 1]);
                const float2 sv = make_float2(sn[16 * rnd + j], sn[16 * rnd + j + 1]);
                float2 r0, r1;
                rope_apply2<kHF>(make_float2(ylo[j], ylo[j + 1]), make_float2(yhi[j], yhi[j + 1]), c, sv, r0, r1);
                ylo[j] = r0.x;
                ylo[j + 1] = r0.y;
                yhi[j] = r1.x;
                yhi[j + 1] = r1.y;
              }
            } else if (!kV) {
              // target RoPE on pairs (c, c + 1): channels c_lo + j, c_lo + j + 1 of ylo (slot
              // 8 rnd + j / 2) and of yhi (slot 16 + 8 rnd + j / 2), two pairs per step
#pragma unroll
              for (int j = 0; j < 16; j += 4) {
#pragma unroll
                for (int hv = 0; hv < 2; ++hv) {
                  float* y = hv ? yhi : ylo;
                  const int m = 16 * hv + 8 * rnd + j / 2;
                  float2 r0, r1;
                  rope_apply2<kHF>(make_float2(y[j], y[j + 2]), make_float2(y[j + 1], y[j + 3]),
                                   make_float2(cs[m], cs[m + 1]), make_float2(sn[m], sn[m + 1]), r0, r1);
                  y[j] = r0.x;
                  y[j + 2] = r0.y;
                  y[j + 1] = r1.x;
                  y[j + 3] = r1.y;
                }
              }
            }
            uint4 v[4];
            v[0] = make_uint4(pack_bf16x2(ylo[0], ylo[1]), pack_bf16x2(ylo[2], ylo[3]), pack_bf16x2(ylo[4], ylo[5]),
                              pack_bf16x2(ylo[6], ylo[7]));
            v[1] = make_uint4(pack_bf16x2(ylo[8], ylo[9]), pack_bf16x2(ylo[10], ylo[11]),
                              pack_bf16x2(ylo[12], ylo[13]), pack_bf16x2(ylo[14], ylo[15]));
            v[2] = make_uint4(pack_bf16x2(yhi[0], yhi[1]), pack_bf16x2(yhi[2], yhi[3]), pack_bf16x2(yhi[4], yhi[5]),
                              pack_bf16x2(yhi[6], yhi[7]));
            v[3] = make_uint4(pack_bf16x2(yhi[8], yhi[9]), pack_bf16x2(yhi[10], yhi[11]),
                              pack_bf16x2(yhi[12], yhi[13]), pack_bf16x2(yhi[14], yhi[15]));
            if (warp_tma || A.paged) {
              // two 32-row x 64-byte pieces (channels 32g.. and 64+32g..), 64-byte swizzle:
              // 16-byte chunk index XOR (row / 2) % 4
              const int sw = (lane >> 1) & 3;
              uint8_t* prow = sb + lane * 64;
              *reinterpret_cast<uint4*>(prow + (((2 * rnd) ^ sw) << 4)) = v[0];
              *reinterpret_cast<uint4*>(prow + (((2 * rnd + 1) ^ sw) << 4)) = v[1];
              *reinterpret_cast<uint4*>(prow + kPieceBytes + (((2 * rnd) ^ sw) << 4)) = v[2];
              *reinterpret_cast<uint4*>(prow + kPieceBytes + (((2 * rnd + 1) ^ sw) << 4)) = v[3];
            } else if (valid) {
              __nv_bfloat16* out = dst + static_cast<int64_t>(l) * A.ts[0] + row_off;
              st_global_hint(out + c_lo, v[0], st_pol);
              st_global_hint(out + c_lo + 8, v[1], st_pol);
              st_global_hint(out + 64 + c_lo, v[2], st_pol);
              st_global_hint(out + 64 + c_lo + 8, v[3], st_pol);
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&bias_empty[bslot]));
          if (A.paged) {
            // Paged rows leave the staging buffer in 64-byte pieces: in store i lanes 8m ..
            // 8m + 7 write row 4i + m, lanes 4 apart the two pieces (channels 32g.. and
            // 64 + 32g..), so each group of four lanes writes one whole 64-byte piece.  The
            // row's block offset comes from the lane that owns the row.
            const int64_t lay_off = static_cast<int64_t>(l) * A.ts[0];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int rr = 4 * i + (lane >> 3);
              const int piece = (lane >> 2) & 1, chunk = lane & 3;
              const uint32_t off_lo = __shfl_sync(0xffffffffu, static_cast<uint32_t>(row_off), rr);
              const uint32_t off_hi = __shfl_sync(0xffffffffu, static_cast<uint32_t>(static_cast<uint64_t>(row_off) >> 32), rr);
              const int ok_row = __shfl_sync(0xffffffffu, valid ? 1 : 0, rr);
              const int sw = (rr >> 1) & 3;
              const uint4 v = *reinterpret_cast<const uint4*>(sb + rr * 64 + piece * kPieceBytes + ((chunk ^ sw) << 4));
              if (ok_row) {
                const int64_t roff = static_cast<int64_t>((static_cast<uint64_t>(off_hi) << 32) | off_lo);
                st_global_hint(dst + lay_off + roff + 64 * piece + 32 * g + 8 * chunk, v, st_pol);
              }
            }
            __syncwarp();   // the staging buffer is read before the next layer writes it
          } else {
            // every contiguous-target layer commits one bulk group per warp (empty when the
            // warp wrote its rows directly), so the group count above identifies the buffer
            if (warp_tma) {
              fence_proxy_async_smem();
              __syncwarp();
            }
            if (lane == 0) {
              if (warp_tma && un.t0 + 32 * q < A.T) {   // skip a box wholly past the sequence end
                // one box: both 32-row x 32-channel pieces (channels 32g.. and 64 + 32g..)
                const int bh = P.out_bh == 2 ? un.b * H + un.h : un.h;
                tma_store_5d(tm_out, smem_u32(sb), 32 * g, un.t0 + 32 * q, 0, bh, l);
              }
              bulk_commit_group();
            }
          }
        }
      };
      if (un.kv) layers(std::true_type{});
      else layers(std::false_type{});
    }
    if (!A.paged && lane == 0) bulk_wait_all();   // this warp's stores are complete
  } else {
    setmaxnreg_inc<kRegsPro>();
    // -------------------------------------------------------- prologue warps ------
    // Thread (quarter q, lane) owns token row r = 32q + lane (TMEM lane r) and all 64 RoPE
    // pairs.  For every load of the schedule, in order: landing buffer -> registers ->
    // (keys) strip the source RoPE in fp32, round to bf16 -> tcgen05.st into the tile's
    // TMEM slot.  These warps run ahead of the epilogue, limited only by the landing
    // buffers and by the release of each slot's previous tile.
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    uint32_t gl = 0, tl_loaded = 0, tfree_par = 0;
    float cs[64], sn[64];   // cos / sin of the source angle of pair i of row r
    bool ok = true;
    for (int u = unit0; ok && u < n_units; u += unit_step) {
      const Unit un = decode_unit(u, H, A.B, tiles, rank);
      if (un.kv == 0) {
        // a row past the sequence end or at an out-of-range position (which the epilogue
        // reports) is rotated by angle 0: its output is never written
        const int t = un.t0 + r;
        int p = t < A.T ? __ldg(&A.pos[static_cast<int64_t>(un.b) * A.T + t]) : 0;
        if (p < 0 || p >= (1 << 24)) p = 0;
#pragma unroll
        for (int i = 0; i < 64; ++i) {
          if constexpr (kHF) {
            sincosf(__fmul_rn(static_cast<float>(p), P.rope.ws_hi[i]), &sn[i], &cs[i]);
            sn[i] = bf16_round(sn[i]);
            cs[i] = bf16_round(cs[i]);
          } else {
            rope_sincos(p, P.rope.ws_hi[i], P.rope.ws_lo[i], P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi,
                        &sn[i], &cs[i]);
          }
        }
      }
      for (int e = 0; ok && e < P.n_loads; ++e) {
        // load word: slot | 4 << i if issuer i used the slot's previous tile (wait for its
        // release) | 16 << i if issuer i uses this tile (signal tready[slot][i])
        const uint32_t lw = static_cast<uint32_t>(__ldg(&P.load_slot[e]));
        const int s = static_cast<int>(lw & 3u);
        const int lb = gl % kLand;
        bool w_ok =
            wait_bar(smem_u32(&land_full[lb]), (gl / kLand) & 1u, abort_flag, P.status, KVX_ERR_TIMEOUT, P.timeout_ns);
        if ((tl_loaded >> s) & 1u) {
#pragma unroll
          for (int i = 0; i < kIssuers; ++i) {
            if (!((lw >> (2 + i)) & 1u)) continue;
            const int bi = s * kIssuers + i;
            w_ok = w_ok && wait_bar(smem_u32(&tfree[bi]), (tfree_par >> bi) & 1u, abort_flag, P.status,
                                    KVX_ERR_TIMEOUT, P.timeout_ns);
            tfree_par ^= 1u << bi;
          }
        }
        if (!__all_sync(0xffffffffu, w_ok)) {
          ok = false;
          break;
        }
        tc_fence_after();
        tl_loaded |= 1u << s;
        const uint8_t* row = land + static_cast<size_t>(lb) * kLandBytes + r * 128;
        const uint32_t scol = tmem_base + lane_addr + kSlotCol0 + s * 64;
#pragma unroll
        for (int c = 0; c < 4; ++c) {   // features 16c .. 16c+15 (a) and 64 + 16c .. 64 + 16c+15 (b)
          uint32_t wa[8], wb[8];
#pragma unroll
          for (int ci = 0; ci < 2; ++ci) {
            const int phys = ((2 * c + ci) ^ (r & 7)) << 4;
            const uint4 va = *reinterpret_cast<const uint4*>(row + phys);
            const uint4 vb = *reinterpret_cast<const uint4*>(row + kHalfBytes + phys);
            wa[4 * ci] = va.x;
            wa[4 * ci + 1] = va.y;
            wa[4 * ci + 2] = va.z;
            wa[4 * ci + 3] = va.w;
            wb[4 * ci] = vb.x;
            wb[4 * ci + 1] = vb.y;
            wb[4 * ci + 2] = vb.z;
            wb[4 * ci + 3] = vb.w;
          }
          if (un.kv == 0 && !kIL) {
#pragma unroll
            for (int w = 0; w < 8; ++w) {   // pairs 16c + 2w and 16c + 2w + 1: (f, f + 64)
              const int m0 = 16 * c + 2 * w, m1 = m0 + 1;
              float2 ra, rb;
              rope_strip2<kHF>(make_float2(bf16_lo(wa[w]), bf16_hi(wa[w])), make_float2(bf16_lo(wb[w]), bf16_hi(wb[w])),
                               make_float2(cs[m0], cs[m1]), make_float2(sn[m0], sn[m1]), ra, rb);
              wa[w] = pack_bf16x2(ra.x, ra.y);
              wb[w] = pack_bf16x2(rb.x, rb.y);
            }
          } else if (un.kv == 0) {
#pragma unroll
            for (int w = 0; w < 8; ++w) {   // pairs 8c + w (word wa[w]) and 32 + 8c + w (word wb[w]): (f, f + 1)
              const int m0 = 8 * c + w, m1 = 32 + 8 * c + w;
              float2 r0, r1;
              rope_strip2<kHF>(make_float2(bf16_lo(wa[w]), bf16_lo(wb[w])), make_float2(bf16_hi(wa[w]), bf16_hi(wb[w])),
                               make_float2(cs[m0], cs[m1]), make_float2(sn[m0], sn[m1]), r0, r1);
              wa[w] = pack_bf16x2(r0.x, r1.x);
              wb[w] = pack_bf16x2(r0.y, r1.y);
            }
          }
          tmem_st_x8(scol + 8 * c, wa);        // TMEM columns 8c .. 8c+7
          tmem_st_x8(scol + 32 + 8 * c, wb);   // TMEM columns 32 + 8c .. 32 + 8c+7
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(smem_u32(&land_empty[lb]));
#pragma unroll
          for (int i = 0; i < kIssuers; ++i)
            if ((lw >> (4 + i)) & 1u) mbar_arrive_cluster(mapa_shared(smem_u32(&tready[s * kIssuers + i]), 0));
        }
        ++gl;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();   // no arrival or MMA of either CTA still targets the other
  tc_fence_after();
  if (warp == 1) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kTmemCols)
                 : "memory");
  }
}

// ------------------------------------------------------------------- host side --

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Belady schedule of source-tile loads over the use sequence (l, j), l-major, into
// kTSlots TMEM slots: the victim is the resident tile whose next use is farthest away;
// among equals, the one whose last use is earliest.  Use (l, j) is issued by issuer l % 2.
// Before a tile is overwritten, every issuer that read it releases the slot (a commit
// after its last use of the tile) and the prologue warps wait for exactly those
// releases.  The final tiles of a unit are released for the first loads of the next one.
// All waits follow the (l, j) order, and with k <= kTSlots a victim always exists, so
// every wait ends.
//   use_flags:  1 first use of the tile by its issuer (wait for tready[slot][issuer]),
//               4 release the slot after the use
//   load_slot:  slot | 4 << i if issuer i must release the slot's previous tile first
//               | 16 << i if issuer i uses the tile (the prologue signals its tready)
void build_plan(const int32_t* sel, int Ls, int Lt, int k, TcPlan* plan) {
  const int n_uses = Lt * k, S = kTSlots;
  std::vector<int> src(n_uses), next_use(n_uses);
  for (int u = 0; u < n_uses; ++u) src[u] = sel[u];
  std::vector<int> seen(Ls, INT_MAX);
  for (int u = n_uses - 1; u >= 0; --u) {
    next_use[u] = seen[src[u]];
    seen[src[u]] = u;
  }
  plan->n_slots = S;
  plan->load_layer.clear();
  plan->load_slot.clear();
  plan->load_first_use.clear();
  plan->use_slot.assign(n_uses, -1);
  plan->use_flags.assign(n_uses, 0);
  std::vector<int> slot_src(S, -1), slot_next(S, INT_MAX), slot_last(S, -1), slot_load(S, -1), slot_first_load(S, -1);
  std::vector<int> last_by(S * kIssuers, -1);   // [slot][issuer] last use of the current tile
  for (int u = 0; u < n_uses; ++u) {
    const int l = u / k, iss = l % kIssuers;
    int s = -1;
    for (int i = 0; i < S; ++i)
      if (slot_src[i] == src[u]) s = i;
    if (s < 0) {
      int best = -1;
      for (int i = 0; i < S; ++i) {
        if (slot_src[i] < 0) {
          best = i;
          break;
        }
        if (best < 0 || slot_next[i] > slot_next[best] ||
            (slot_next[i] == slot_next[best] && slot_last[i] < slot_last[best]))
          best = i;
      }
      s = best;
      int word = s;
      for (int i = 0; i < kIssuers; ++i) {
        const int lu = last_by[s * kIssuers + i];
        if (lu >= 0) {
          plan->use_flags[lu] |= 4;
          word |= 4 << i;
        }
        last_by[s * kIssuers + i] = -1;
      }
      if (slot_first_load[s] < 0) slot_first_load[s] = static_cast<int>(plan->load_slot.size());
      plan->load_layer.push_back(src[u]);
      plan->load_slot.push_back(word);
      plan->load_first_use.push_back(l);
      slot_src[s] = src[u];
      slot_load[s] = static_cast<int>(plan->load_slot.size()) - 1;
    }
    if (last_by[s * kIssuers + iss] < 0) {
      plan->use_flags[u] |= 1;
      plan->load_slot[slot_load[s]] |= 16 << iss;
    }
    last_by[s * kIssuers + iss] = u;
    plan->use_slot[u] = s;
    slot_next[s] = next_use[u];
    slot_last[s] = u;
  }
  for (int s = 0; s < S; ++s) {
    if (slot_src[s] < 0) continue;
    for (int i = 0; i < kIssuers; ++i) {
      const int lu = last_by[s * kIssuers + i];
      if (lu >= 0) {
        plan->use_flags[lu] |= 4;
        plan->load_slot[slot_first_load[s]] |= 4 << i;
      }
    }
  }
  plan->n_loads = static_cast<int>(plan->load_layer.size());
}

// The issuers' 5-bit word of use u: slot | 4 first use of the tile by its issuer | 16
// release the slot after the use.
uint32_t use_bits(const TcPlan& p, int u) {
  return static_cast<uint32_t>(p.use_slot[u]) | ((p.use_flags[u] & 1) ? 4u : 0u) | ((p.use_flags[u] & 4) ? 16u : 0u);
}

}  // namespace

void* tensor_map_encoder() { return reinterpret_cast<void*>(get_encode()); }

bool tc_supported(const kvx_ctx* c, std::string* why) {
  std::string w;
  if (c->cache_dtype != KVX_BF16) w = "needs bf16 caches";
  else if (c->d != kD) w = "needs head_dim 128";
  else if (c->head_mix != KVX_PER_HEAD) w = "needs per-head features";
  else if (c->k > kTSlots) w = "needs k <= 4 (one target layer's source tiles must fit in tensor memory)";
  else if (static_cast<int64_t>(c->Lt) * 2 * c->H * kD > INT_MAX) w = "too many W rows";
  if (why) *why = w;
  return w.empty();
}

kvx_status repack_wt(kvx_ctx* c, const void* W_host, size_t F) {
  // W [L_t][2][H][F][128] -> W^T [L_t][2][H][128][F] (B operand, K-major)
  const size_t blocks = static_cast<size_t>(c->Lt) * 2 * c->H;
  std::vector<uint16_t> wt(blocks * F * kD);
  const uint16_t* w = static_cast<const uint16_t*>(W_host);
  for (size_t blk = 0; blk < blocks; ++blk) {
    const uint16_t* srcb = w + blk * F * kD;
    uint16_t* dstb = wt.data() + blk * F * kD;
    for (size_t f = 0; f < F; ++f)
      for (int n = 0; n < kD; ++n) dstb[static_cast<size_t>(n) * F + f] = srcb[f * kD + n];
  }
  cudaError_t e = cudaMalloc(&c->d_Wt, wt.size() * 2);
  if (e != cudaSuccess) {
    set_error(std::string("kvx_create: cudaMalloc W^T: ") + cudaGetErrorString(e));
    return KVX_ERR_OOM;
  }
  if ((e = cudaMemcpy(c->d_Wt, wt.data(), wt.size() * 2, cudaMemcpyHostToDevice)) != cudaSuccess) {
    set_error(std::string("kvx_create: upload W^T: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

kvx_status tc_prepare(kvx_ctx* c, const void* W_host) {
  kvx_status st = c->weight_dtype == KVX_F32 ? repack_wt_hilo(c, W_host, c->F) : repack_wt(c, W_host, c->F);
  if (st != KVX_OK) return st;
  cudaError_t e;
  build_plan(c->sel.data(), c->Ls, c->Lt, c->k, &c->plan);
  c->plan.n_wst = kNW;   // two rings of kRing stages
  c->plan.n_land = kLand;
  const TcPlan& p = c->plan;
  // per target layer, one word: 5 bits per use j (slot | 4 first use by its issuer |
  // 16 release after)
  std::vector<int32_t> pack(c->Lt, 0);
  for (int l = 0; l < c->Lt; ++l)
    for (int j = 0; j < c->k; ++j) {
      const int u = l * c->k + j;
      pack[l] |= static_cast<int32_t>(use_bits(p, u) << (5 * j));
    }
  std::vector<int32_t> tab;
  tab.insert(tab.end(), p.load_layer.begin(), p.load_layer.end());
  tab.insert(tab.end(), p.load_slot.begin(), p.load_slot.end());
  tab.insert(tab.end(), p.load_first_use.begin(), p.load_first_use.end());
  tab.insert(tab.end(), pack.begin(), pack.end());
  if ((e = cudaMalloc(&c->d_plan, tab.size() * 4)) != cudaSuccess) {
    set_error(std::string("kvx_create: cudaMalloc plan: ") + cudaGetErrorString(e));
    return KVX_ERR_OOM;
  }
  if ((e = cudaMemcpy(c->d_plan, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice)) != cudaSuccess) {
    set_error(std::string("kvx_create: upload plan: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

kvx_status launch_tc(const kvx_ctx* c, const MapArgs& a, cudaStream_t stream) {
  auto encode = get_encode();
  if (!encode) {
    set_error("kvx_map: cuTensorMapEncodeTiled unavailable");
    return KVX_ERR_CUDA;
  }
  TcParams P;
  std::memset(&P, 0, sizeof(P));
  const cuuint32_t ones[5] = {1, 1, 1, 1, 1};
  // source maps: dims (d, T, H, B, L_s), strides in bytes for dims 1..4
  const cuuint64_t sdims[5] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(a.T),
                               static_cast<cuuint64_t>(c->H), static_cast<cuuint64_t>(a.B),
                               static_cast<cuuint64_t>(c->Ls)};
  const cuuint64_t sstr[4] = {static_cast<cuuint64_t>(a.ss[3]) * 2, static_cast<cuuint64_t>(a.ss[2]) * 2,
                              static_cast<cuuint64_t>(a.ss[1]) * 2, static_cast<cuuint64_t>(a.ss[0]) * 2};
  const cuuint32_t box[5] = {64, kTileM, 1, 1, 1};
  for (int kv = 0; kv < 2; ++kv) {
    CUresult r = encode(kv ? &P.tm_v : &P.tm_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                        const_cast<void*>(kv ? a.src_v : a.src_k), sdims, sstr, box, ones,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      set_error("kvx_map: source tensor map rejected (strides or sizes)");
      return KVX_ERR_UNSUPPORTED;
    }
  }
  // Target maps for the per-warp TMA stores: dims (64 channels, T, 2 halves, heads, L_t),
  // so that one box (32 channels x 32 rows x both halves, 4 KB) holds a warp's share of a
  // layer.  The inner box extent equals the 64-byte swizzle span.  The batch folds into
  // the head dim when B = 1 or the batch stride is H head strides; other contiguous layouts
  // take direct stores.
  P.out_bh = 0;
  if (!a.paged && (a.B == 1 || a.ts[1] == static_cast<int64_t>(c->H) * a.ts[2])) {
    P.out_bh = a.B == 1 ? 1 : 2;
    const cuuint32_t tbox[5] = {32, 32, 2, 1, 1};
    const cuuint64_t tdims[5] = {64, static_cast<cuuint64_t>(a.T), 2,
                                 static_cast<cuuint64_t>(c->H) * static_cast<cuuint64_t>(a.B),
                                 static_cast<cuuint64_t>(c->Lt)};
    const cuuint64_t tstr[4] = {static_cast<cuuint64_t>(a.ts[3]) * 2, 64 * 2, static_cast<cuuint64_t>(a.ts[2]) * 2,
                                static_cast<cuuint64_t>(a.ts[0]) * 2};
    for (int kv = 0; kv < 2; ++kv) {
      CUresult r = encode(kv ? &P.tm_out_v : &P.tm_out_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                          kv ? a.tgt_v : a.tgt_k, tdims, tstr, tbox, ones, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS) {
        set_error("kvx_map: target tensor map rejected (strides or sizes)");
        return KVX_ERR_UNSUPPORTED;
      }
    }
  }
  // fp32 weights: W^T holds [W_hi | W_lo], 2F columns
  const cuuint64_t wcols = static_cast<cuuint64_t>(c->F) * (c->weight_dtype == KVX_F32 ? 2 : 1);
  const cuuint64_t wdims[2] = {wcols, static_cast<cuuint64_t>(c->Lt) * 2 * c->H * kD};
  const cuuint64_t wstr[1] = {wcols * 2};
  const cuuint32_t wbox[2] = {64, kD / 2};   // one CTA's 64 output rows x 64 features
  CUresult r = encode(&P.tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->d_Wt, wdims, wstr, wbox, ones,
                      CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("kvx_map: weight tensor map rejected");
    return KVX_ERR_CUDA;
  }
  const TcPlan& p = c->plan;
  P.a = a;
  P.load_layer = c->d_plan;
  P.load_slot = c->d_plan + p.n_loads;
  P.use_pack = reinterpret_cast<const uint32_t*>(c->d_plan + 3 * p.n_loads);
  P.bias = c->d_b;
  P.status = c->d_status;
  P.Lt = c->Lt;
  P.H = c->H;
  P.k = c->k;
  P.n_loads = p.n_loads;
  // work units are pairs of adjacent 128-token tiles (one per CTA of a cluster)
  P.tiles_per_seq = (a.T + 2 * kTileM - 1) / (2 * kTileM);
  const int64_t units = static_cast<int64_t>(a.B) * P.tiles_per_seq * c->H * 2;
  if (units > INT_MAX) {
    set_error("kvx_map: too many work units");
    return KVX_ERR_UNSUPPORTED;
  }
  P.n_units = static_cast<int>(units);
  P.rope = c->rope;
  P.timeout_ns = c->wait_limit_ns ? c->wait_limit_ns : kTimeoutNs;
  P.skip_bias = static_cast<int32_t>(c->skip_bias_row);
  const size_t smem = smem_bytes();
  const bool hf = c->rope_numerics == KVX_ROPE_HF;
  const bool il = c->rope_style == KVX_ROPE_INTERLEAVED;
  void (*const kernels[8])(TcParams) = {tc_map_kernel<false, 1, false>, tc_map_kernel<true, 1, false>,
                                        tc_map_kernel<false, 2, false>, tc_map_kernel<true, 2, false>,
                                        tc_map_kernel<false, 1, true>,  tc_map_kernel<true, 1, true>,
                                        tc_map_kernel<false, 2, true>,  tc_map_kernel<true, 2, true>};
  void (*kernel)(TcParams) = kernels[(il ? 4 : 0) + (c->weight_dtype == KVX_F32 ? 2 : 0) + (hf ? 1 : 0)];
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: smem attribute: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  // The warpgroups' register shares (setmaxnreg) are drawn from what the launch holds: a
  // build that launched with fewer registers per thread would leave an increase waiting.
  cudaFuncAttributes fa;
  e = cudaFuncGetAttributes(&fa, kernel);
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: kernel attributes: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  if (static_cast<uint32_t>(fa.numRegs) * kThreads < kRegsCtl * 128 + kRegsEpi * 256 + kRegsPro * 128) {
    set_error("kvx_map: tensor-core kernel built with " + std::to_string(fa.numRegs) +
              " registers per thread, too few for its warpgroup register split");
    return KVX_ERR_UNSUPPORTED;
  }
  const int grid = 2 * static_cast<int>(std::min<int64_t>(units, std::max(c->sm_count / 2, 1)));   // CTA pairs
  kernel<<<grid, kThreads, smem, stream>>>(P);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: tensor-core launch: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

}  // namespace kvx

extern "C" {

KVX_API kvx_status kvx_tc_load_schedule(const int32_t* selection, int32_t src_layers, int32_t tgt_layers, int32_t k,
                                        int32_t* n_loads, int32_t* load_layer, int32_t* load_word,
                                        int32_t* use_word) {
  kvx::set_error("");
  auto fail = [](kvx_status s, const char* m) {
    kvx::set_error(m);
    return s;
  };
  if (!selection || !n_loads || !load_layer || !load_word || !use_word)
    return fail(KVX_ERR_INVALID_ARG, "kvx_tc_load_schedule: NULL argument");
  if (src_layers < 1 || tgt_layers < 1 || k < 1 || k > src_layers)
    return fail(KVX_ERR_INVALID_ARG, "kvx_tc_load_schedule: need src_layers, tgt_layers >= 1 and k in [1, src_layers]");
  if (k > kvx::kTSlots)
    return fail(KVX_ERR_UNSUPPORTED, "kvx_tc_load_schedule: the per-head tensor-core kernel holds at most 4 source tiles");
  for (int32_t l = 0; l < tgt_layers; ++l) {
    const int32_t* row = selection + static_cast<size_t>(l) * k;
    for (int32_t j = 0; j < k; ++j) {
      if (row[j] < 0 || row[j] >= src_layers)
        return fail(KVX_ERR_INVALID_ARG, "kvx_tc_load_schedule: selection entry outside [0, src_layers)");
      for (int32_t i = 0; i < j; ++i)
        if (row[i] == row[j]) return fail(KVX_ERR_INVALID_ARG, "kvx_tc_load_schedule: duplicate source layer in a row");
    }
  }
  kvx::TcPlan plan;
  kvx::build_plan(selection, src_layers, tgt_layers, k, &plan);
  *n_loads = plan.n_loads;
  for (int e = 0; e < plan.n_loads; ++e) {
    load_layer[e] = plan.load_layer[e];
    load_word[e] = plan.load_slot[e];
  }
  for (int u = 0; u < tgt_layers * k; ++u) use_word[u] = static_cast<int32_t>(kvx::use_bits(plan, u));
  return KVX_OK;
}

}  // extern "C"
