// Tensor-core mapping kernel for sm_103a (tcgen05 + TMEM + TMA), bf16 caches and
// weights, head_dim 128, per-head features, half-split RoPE pairs.
//
// What it computes is Eq. ridge_kv with the Sec. 3.3 RoPE composition:
//   K_t^{l,h} = R_t(t) ( [R_s(t)^-1 K_s^{sel[l][j]}[h]]_j W_K^{l,h} + b_K^{l,h} ),
//   V_t^{l,h} =          [V_s^{sel[l][j]}[h]]_j W_V^{l,h} + b_V^{l,h},
// with the stripped keys rounded to bf16 before the contraction and fp32 accumulation.
//
// Work unit = (sequence b, 128-token tile, head h, K|V).  A persistent CTA walks all
// target layers of a unit.  The k source tiles a target layer concatenates are
// 128 x 128 bf16 tiles in shared memory; a host-built schedule (Belady over the
// sequence of (layer, j) uses) keeps every source tile resident for as long as later
// target layers select it, so each source layer is read from HBM once per token tile
// and shared by all target layers that select it (Sec. 3.2 selection is near
// proportional depth, so a ring of k+1 slots almost never reloads).
//
// The contraction of target layer l is the GEMM D[128 tok x 128 ch] = X[128 x kd] W[kd x 128]
// on tcgen05 (cta_group::1, M = N = 128, K = 16 per instruction), A = source slots
// (K-major, 128-byte swizzle, as TMA lands them), B = W^T streamed through a ring of
// 16 KB stages (128 output channels x 64 features), D = fp32 in TMEM, double buffered.
//
// Warp roles (384 threads):
//   warp 0      TMA producer of source tiles (one thread)
//   warp 1      MMA issuer (one thread)
//   warp 2      TMEM allocator
//   warp 3      TMA producer of W stages (one thread)
//   warps 4-11  two "transform" warpgroups.  Thread (group g, row r) owns token row r
//               (= TMEM lane r) and RoPE pairs i in [32g, 32g+32) (channels i, i+64):
//               it strips the source RoPE from key tiles in place (fp32, round to
//               bf16) and runs the epilogue (TMEM -> registers, + bias, target RoPE for
//               keys, bf16, 16-byte global stores, contiguous or paged).
//
// Every mbarrier wait is bounded: after kTimeoutNs the kernel raises KVX_ERR_TIMEOUT
// in the status word, sets a shared abort flag that every role polls, waits (again
// bounded) for its own TMA copies and MMAs in flight, frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>
#include <vector>

#include "kvx_internal.h"
#include "kvx_rope.cuh"

namespace kvx {
namespace {

constexpr int kThreads = 384;
constexpr int kTileM = 128;                      // tokens per work unit
constexpr int kD = 128;                          // head_dim of this kernel
constexpr uint32_t kSlotBytes = kTileM * kD * 2; // 32 KB: two 64-column SW128 halves
constexpr uint32_t kHalfBytes = kSlotBytes / 2;  // 16 KB
constexpr uint32_t kWStageBytes = 128 * 64 * 2;  // 16 KB: 128 channels x 64 features
constexpr int kMaxSlots = 8;
constexpr int kMaxWStages = 8;
constexpr uint32_t kTmemCols = 256;              // two 128-column fp32 accumulators
constexpr uint64_t kTimeoutNs = 4000000000ull;   // 4 s
constexpr size_t kSmemLimit = 232448;            // 227 KB opt-in per CTA

struct TcParams {
  CUtensorMap tm_k;   // source keys   [L_s][B][H][T][128] bf16, box 64 x 128
  CUtensorMap tm_v;   // source values
  CUtensorMap tm_w;   // W^T           [L_t*2*H*128][F] bf16, box 64 x 128
  MapArgs a;
  const int32_t* load_layer;   // [n_loads]
  const int32_t* load_slot;    // [n_loads]
  const int32_t* load_first;   // [n_loads] first target layer using the load
  const int32_t* use_slot;     // [L_t*k]
  const int32_t* use_flags;    // [L_t*k] bit 0: first use of a load; bit 1: release after
  const float* bias;           // [L_t][2][H][128] fp32
  int32_t* status;
  int32_t Lt, H, k, n_slots, n_wst, n_loads, tiles_per_seq, n_units, same_theta;
  RopeTables rope;
};

// ------------------------------------------------------------------ PTX wrappers --

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ uint32_t mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok;
}

__device__ __forceinline__ uint64_t global_timer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait for the phase of the given parity.  false = timed out or aborted.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile uint32_t* abort_flag,
                                         int32_t* status) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0 = 0;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 127u) == 0) {
      if (*abort_flag) return false;
      const uint64_t now = global_timer();
      if (t0 == 0) {
        t0 = now;
      } else if (now - t0 > kTimeoutNs) {
        *abort_flag = 1u;
        atomicCAS(status, 0, KVX_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

// Teardown wait: ignores the abort flag, still bounded in time.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const uint64_t t0 = global_timer();
  while (!mbar_try_wait(bar, parity))
    if (global_timer() - t0 > kTimeoutNs) break;
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int c0,
                                            int c1, int c2, int c3, int c4, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7], %8;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(bar),
      "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int c0,
                                            int c1, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar), "l"(policy)
      : "memory");
}

// L2 prefetch of one tensor-map tile (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_5d(const CUtensorMap* map, int c0, int c1, int c2, int c3, int c4) {
  asm volatile("cp.async.bulk.prefetch.tensor.5d.L2.global.tile [%0, {%1, %2, %3, %4, %5}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4)
               : "memory");
}

__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap* map, int c0, int c1) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1)
               : "memory");
}

// 16-byte global store that bypasses L1 and is marked evict-first in L2 (the target
// cache is written once and not read by this kernel).
__device__ __forceinline__ void st_global_stream(void* ptr, uint4 v, uint64_t policy) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.b32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(ptr),
               "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(policy)
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row core groups 1024 B
// apart (stride byte offset), leading byte offset unused for this layout (1), descriptor
// version 1 (bits 46-47), swizzle mode 2 = 128B (bits 61-63).  Tiles are 1024-aligned.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return static_cast<uint64_t>((saddr >> 4) & 0x3FFFu) | (static_cast<uint64_t>(1) << 16) |
         (static_cast<uint64_t>(1024 >> 4) << 32) | (static_cast<uint64_t>(1) << 46) |
         (static_cast<uint64_t>(2) << 61);
}

// Instruction descriptor, kind::f16: D fp32 (bit 4), A bf16 (bits 7-9 = 1), B bf16 (bits
// 10-12 = 1), both K-major, N >> 3 at bits 17-22, M >> 4 at bits 24-28.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

// Two 16-column TMEM loads (32 lanes x 32 bit each) and the wait, in one asm block so
// the registers are complete when it returns.
__device__ __forceinline__ void tmem_ld_2x16(uint32_t taddr_lo, uint32_t taddr_hi, uint32_t (&lo)[16],
                                             uint32_t (&hi)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%32];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%33];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(lo[0]), "=r"(lo[1]), "=r"(lo[2]), "=r"(lo[3]), "=r"(lo[4]), "=r"(lo[5]), "=r"(lo[6]),
        "=r"(lo[7]), "=r"(lo[8]), "=r"(lo[9]), "=r"(lo[10]), "=r"(lo[11]), "=r"(lo[12]), "=r"(lo[13]),
        "=r"(lo[14]), "=r"(lo[15]), "=r"(hi[0]), "=r"(hi[1]), "=r"(hi[2]), "=r"(hi[3]), "=r"(hi[4]),
        "=r"(hi[5]), "=r"(hi[6]), "=r"(hi[7]), "=r"(hi[8]), "=r"(hi[9]), "=r"(hi[10]), "=r"(hi[11]),
        "=r"(hi[12]), "=r"(hi[13]), "=r"(hi[14]), "=r"(hi[15])
      : "r"(taddr_lo), "r"(taddr_hi)
      : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ void report(int32_t* status, int code) { atomicCAS(status, 0, code); }

struct Unit {
  int b, t0, h, kv;
};

// Units are visited u = blockIdx.x + i * gridDim.x.  With an even grid, u & 1 would pin
// every CTA to K or to V units; flipping it every round makes each CTA alternate, which
// balances the (heavier) key units across CTAs.  u and u ^ 1 share u / grid, so the
// mapping stays a bijection.
__device__ __forceinline__ Unit decode_unit(int u, int H, int tiles) {
  Unit r;
  r.kv = (u & 1) ^ ((gridDim.x & 1) ? 0 : static_cast<int>((u / gridDim.x) & 1));
  int rest = u >> 1;
  r.h = rest % H;
  rest /= H;
  r.t0 = (rest % tiles) * kTileM;
  r.b = rest / tiles;
  return r;
}

// ------------------------------------------------------------------------ kernel --

__global__ void __launch_bounds__(kThreads, 1) tc_map_kernel(const __grid_constant__ TcParams P) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = P.n_slots, NW = P.n_wst;
  uint8_t* slots = smem;
  uint8_t* wst = smem + static_cast<size_t>(S) * kSlotBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(wst + static_cast<size_t>(NW) * kWStageBytes);
  uint64_t* full = bars;                  // [S] TMA landed
  uint64_t* ready = full + S;             // [S] keys stripped (K units)
  uint64_t* empty = ready + S;            // [S] slot released by the MMA
  uint64_t* wfull = empty + S;            // [NW]
  uint64_t* wempty = wfull + NW;          // [NW]
  uint64_t* accf = wempty + NW;           // [2]
  uint64_t* acce = accf + 2;              // [2]
  uint64_t* drain = acce + 2;             // [1]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  volatile uint32_t* abort_flag = tmem_holder + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&ready[s]), 8);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int s = 0; s < NW; ++s) {
      mbar_init(smem_u32(&wfull[s]), 1);
      mbar_init(smem_u32(&wempty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&accf[a]), 1);
      mbar_init(smem_u32(&acce[a]), 8);
    }
    mbar_init(smem_u32(drain), 1);
    *abort_flag = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_holder)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const int Lt = P.Lt, k = P.k, H = P.H;
  const int n_units = P.n_units, tiles = P.tiles_per_seq;
  const MapArgs& A = P.a;

  if (warp == 0) {
    // ------------------------------------------------ source-tile producer --------
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t loaded = 0, empty_par = 0, full_cnt_par = 0;
      bool ok = true;
      constexpr int kPrefetch = 4;   // source tiles pulled into L2 ahead of their TMA load
      auto prefetch = [&](int u, int e) {
        if (e >= P.n_loads) {
          e -= P.n_loads;
          u += gridDim.x;
        }
        if (u >= n_units) return;
        const Unit pu = decode_unit(u, H, tiles);
        const CUtensorMap* ptm = pu.kv ? &P.tm_v : &P.tm_k;
        const int L = __ldg(&P.load_layer[e]);
        tma_prefetch_5d(ptm, 0, pu.t0, pu.h, pu.b, L);
        tma_prefetch_5d(ptm, 64, pu.t0, pu.h, pu.b, L);
      };
      if (blockIdx.x < n_units)
        for (int e = 0; e < kPrefetch && e < P.n_loads; ++e) prefetch(blockIdx.x, e);
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        const Unit un = decode_unit(u, H, tiles);
        const CUtensorMap* tm = un.kv ? &P.tm_v : &P.tm_k;
        for (int e = 0; e < P.n_loads; ++e) {
          const int s = __ldg(&P.load_slot[e]);
          const int L = __ldg(&P.load_layer[e]);
          prefetch(u, e + kPrefetch);
          if ((loaded >> s) & 1u) {
            if (!wait_bar(smem_u32(&empty[s]), (empty_par >> s) & 1u, abort_flag, P.status)) {
              ok = false;
              break;
            }
            empty_par ^= 1u << s;
          }
          const uint32_t dst = smem_u32(slots + static_cast<size_t>(s) * kSlotBytes);
          mbar_expect_tx(smem_u32(&full[s]), kSlotBytes);
          tma_load_5d(dst, tm, smem_u32(&full[s]), 0, un.t0, un.h, un.b, L, pol);
          tma_load_5d(dst + kHalfBytes, tm, smem_u32(&full[s]), 64, un.t0, un.h, un.b, L, pol);
          loaded |= 1u << s;
          full_cnt_par ^= 1u << s;
        }
      }
      if (!ok) {  // wait for the copies still in flight into each slot
        for (int s = 0; s < S; ++s)
          if ((loaded >> s) & 1u) drain_wait(smem_u32(&full[s]), ((full_cnt_par >> s) & 1u) ^ 1u);
      }
    }
  } else if (warp == 3) {
    // ------------------------------------------------------------ W producer ------
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();
      uint32_t wi = 0;
      bool ok = true;
      const int chunks = 2 * k;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        const Unit un = decode_unit(u, H, tiles);
        for (int l = 0; ok && l < Lt; ++l) {
          const int row0 = ((l * 2 + un.kv) * H + un.h) * kD;
          for (int c = 0; c < chunks; ++c, ++wi) {
            const int st = wi % NW;
            const uint32_t round = wi / NW;
            if (round > 0 &&
                !wait_bar(smem_u32(&wempty[st]), (round - 1) & 1u, abort_flag, P.status)) {
              ok = false;
              break;
            }
            // pull the same chunk of the next layer (or of the next unit's layer 0) into L2
            if (l + 1 < Lt) {
              tma_prefetch_2d(&P.tm_w, c * 64, (((l + 1) * 2 + un.kv) * H + un.h) * kD);
            } else if (u + static_cast<int>(gridDim.x) < n_units) {
              const Unit nu = decode_unit(u + gridDim.x, H, tiles);
              tma_prefetch_2d(&P.tm_w, c * 64, (nu.kv * H + nu.h) * kD);
            }
            mbar_expect_tx(smem_u32(&wfull[st]), kWStageBytes);
            tma_load_2d(smem_u32(wst + static_cast<size_t>(st) * kWStageBytes), &P.tm_w,
                        smem_u32(&wfull[st]), c * 64, row0, pol);
          }
        }
      }
      if (!ok) {
        // the last min(wi, NW) stages may still be landing
        const uint32_t first = wi > static_cast<uint32_t>(NW) ? wi - NW : 0;
        for (uint32_t i = first; i < wi; ++i) drain_wait(smem_u32(&wfull[i % NW]), (i / NW) & 1u);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA ---------
    if (lane == 0) {
      constexpr uint32_t idesc = make_idesc(kTileM, kD);
      uint32_t full_par = 0, ready_par = 0, wi = 0, li = 0;
      bool ok = true, issued = false;
      for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
        const Unit un = decode_unit(u, H, tiles);
        for (int l = 0; ok && l < Lt; ++l, ++li) {
          const uint32_t a = li & 1u;
          if (li >= 2 && !wait_bar(smem_u32(&acce[a]), ((li >> 1) - 1) & 1u, abort_flag, P.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + a * kD;
          for (int j = 0; ok && j < k; ++j) {
            const int s = __ldg(&P.use_slot[l * k + j]);
            const int fl = __ldg(&P.use_flags[l * k + j]);
            if (fl & 1) {
              bool w_ok;
              if (un.kv == 0) {
                w_ok = wait_bar(smem_u32(&ready[s]), (ready_par >> s) & 1u, abort_flag, P.status);
                ready_par ^= 1u << s;
              } else {
                w_ok = wait_bar(smem_u32(&full[s]), (full_par >> s) & 1u, abort_flag, P.status);
              }
              full_par ^= 1u << s;
              if (!w_ok) {
                ok = false;
                break;
              }
              tc_fence_after();
            }
            const uint32_t a_base = smem_u32(slots + static_cast<size_t>(s) * kSlotBytes);
            for (int half = 0; half < 2; ++half, ++wi) {
              const int st = wi % NW;
              if (!wait_bar(smem_u32(&wfull[st]), (wi / NW) & 1u, abort_flag, P.status)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t b_base = smem_u32(wst + static_cast<size_t>(st) * kWStageBytes);
#pragma unroll
              for (int kk = 0; kk < 4; ++kk) {
                tc_mma(d_tmem, sw128_desc(a_base + half * kHalfBytes + kk * 32), sw128_desc(b_base + kk * 32),
                       idesc, (j | half | kk) != 0);
              }
              issued = true;
              tc_commit(smem_u32(&wempty[st]));
            }
            if (ok && (fl & 2)) tc_commit(smem_u32(&empty[s]));
          }
          if (ok) tc_commit(smem_u32(&accf[a]));
        }
      }
      // make sure every MMA (and every commit) has completed before TMEM is freed
      if (issued || !ok) {
        tc_commit(smem_u32(drain));
        drain_wait(smem_u32(drain), 0);
      }
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------- transform warps ------
    const int g = (warp - 4) >> 2;          // column group: pairs [32g, 32g+32)
    const int q = warp & 3;                 // TMEM lane quarter
    const int r = q * 32 + lane;            // token row within the tile
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    uint32_t full_par = 0, li = 0;
    float cs[32], sn[32];
    bool ok = true;
    const uint64_t st_pol = policy_evict_first();
    for (int u = blockIdx.x; ok && u < n_units; u += gridDim.x) {
      const Unit un = decode_unit(u, H, tiles);
      const int t = un.t0 + r;
      bool valid = t < A.T;
      int p = 0;
      if (valid) {
        p = __ldg(&A.pos[static_cast<int64_t>(un.b) * A.T + t]);
        if (p < 0 || p >= (1 << 24)) {
          report(P.status, KVX_ERR_DEVICE_BOUNDS);
          valid = false;
          p = 0;
        }
      }
      int64_t row_off = 0;
      if (valid) {
        if (!A.paged) {
          row_off = un.b * A.ts[1] + un.h * A.ts[2] + static_cast<int64_t>(t) * A.ts[3];
        } else {
          const int lb = p / A.block_size;
          const int blk = lb < A.max_blocks ? __ldg(&A.block_table[static_cast<int64_t>(un.b) * A.max_blocks + lb]) : -1;
          if (blk < 0 || blk >= A.n_blocks) {
            report(P.status, KVX_ERR_DEVICE_BOUNDS);
            valid = false;
          } else {
            row_off = static_cast<int64_t>(blk) * A.ts[1] + un.h * A.ts[2] +
                      static_cast<int64_t>(p % A.block_size) * A.ts[3];
          }
        }
      }
      if (un.kv == 0) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          rope_sincos(p, P.rope.wt_hi[32 * g + j], P.rope.wt_lo[32 * g + j], P.rope.two_pi_hi,
                      P.rope.two_pi_lo, P.rope.inv_two_pi, &sn[j], &cs[j]);
      }
      __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(un.kv ? A.tgt_v : A.tgt_k);
      int e = 0;
      for (int l = 0; ok && l < Lt; ++l, ++li) {
        // strip the key tiles that layer l + 1 needs first
        while (e < P.n_loads && __ldg(&P.load_first[e]) <= l + 1) {
          const int s = __ldg(&P.load_slot[e]);
          if (un.kv == 0) {
            const bool w_ok = wait_bar(smem_u32(&full[s]), (full_par >> s) & 1u, abort_flag, P.status);
            if (!__all_sync(0xffffffffu, w_ok)) {
              ok = false;
              break;
            }
            uint8_t* row = slots + static_cast<size_t>(s) * kSlotBytes + r * 128;
#pragma unroll
            for (int c4 = 0; c4 < 4; ++c4) {
              const int phys = ((4 * g + c4) ^ (r & 7)) << 4;
              uint4* pa = reinterpret_cast<uint4*>(row + phys);
              uint4* pb = reinterpret_cast<uint4*>(row + kHalfBytes + phys);
              uint4 va = *pa, vb = *pb;
              uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
              for (int m = 0; m < 4; ++m) {
                float ca0, sa0, ca1, sa1;
                const int j0 = 8 * c4 + 2 * m;
                if (P.same_theta) {
                  ca0 = cs[j0];
                  sa0 = sn[j0];
                  ca1 = cs[j0 + 1];
                  sa1 = sn[j0 + 1];
                } else {
                  rope_sincos(p, P.rope.ws_hi[32 * g + j0], P.rope.ws_lo[32 * g + j0], P.rope.two_pi_hi,
                              P.rope.two_pi_lo, P.rope.inv_two_pi, &sa0, &ca0);
                  rope_sincos(p, P.rope.ws_hi[32 * g + j0 + 1], P.rope.ws_lo[32 * g + j0 + 1],
                              P.rope.two_pi_hi, P.rope.two_pi_lo, P.rope.inv_two_pi, &sa1, &ca1);
                }
                const float a0 = bf16_lo(wa[m]), a1 = bf16_hi(wa[m]);
                const float b0 = bf16_lo(wb[m]), b1 = bf16_hi(wb[m]);
                // rotation by -t*omega: a' = a c + b s, b' = b c - a s
                wa[m] = pack_bf16x2(__fmaf_rn(a0, ca0, __fmul_rn(b0, sa0)), __fmaf_rn(a1, ca1, __fmul_rn(b1, sa1)));
                wb[m] = pack_bf16x2(__fmaf_rn(b0, ca0, -__fmul_rn(a0, sa0)), __fmaf_rn(b1, ca1, -__fmul_rn(a1, sa1)));
              }
              *pa = make_uint4(wa[0], wa[1], wa[2], wa[3]);
              *pb = make_uint4(wb[0], wb[1], wb[2], wb[3]);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&ready[s]));
          }
          full_par ^= 1u << s;
          ++e;
        }
        if (!ok) break;
        // epilogue of layer l
        const uint32_t a = li & 1u;
        const bool w_ok = wait_bar(smem_u32(&accf[a]), (li >> 1) & 1u, abort_flag, P.status);
        if (!__all_sync(0xffffffffu, w_ok)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t col = tmem_base + a * kD + 32 * g;
        const float* bias = P.bias + (static_cast<size_t>(l * 2 + un.kv) * H + un.h) * kD + 32 * g;
        __nv_bfloat16* out = dst + static_cast<int64_t>(l) * A.ts[0] + row_off + 32 * g;
#pragma unroll
        for (int rnd = 0; rnd < 2; ++rnd) {
          uint32_t lo[16], hi[16];
          tmem_ld_2x16(col + 16 * rnd + lane_addr, col + 64 + 16 * rnd + lane_addr, lo, hi);
          if (rnd == 1) {  // the accumulator is free for the next layer's MMAs
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&acce[a]));
          }
          if (valid) {
            float ylo[16], yhi[16];
#pragma unroll
            for (int j = 0; j < 16; j += 4) {
              const float4 b0 = __ldg(reinterpret_cast<const float4*>(bias + 16 * rnd + j));
              const float4 b1 = __ldg(reinterpret_cast<const float4*>(bias + 64 + 16 * rnd + j));
              ylo[j] = __fadd_rn(__uint_as_float(lo[j]), b0.x);
              ylo[j + 1] = __fadd_rn(__uint_as_float(lo[j + 1]), b0.y);
              ylo[j + 2] = __fadd_rn(__uint_as_float(lo[j + 2]), b0.z);
              ylo[j + 3] = __fadd_rn(__uint_as_float(lo[j + 3]), b0.w);
              yhi[j] = __fadd_rn(__uint_as_float(hi[j]), b1.x);
              yhi[j + 1] = __fadd_rn(__uint_as_float(hi[j + 1]), b1.y);
              yhi[j + 2] = __fadd_rn(__uint_as_float(hi[j + 2]), b1.z);
              yhi[j + 3] = __fadd_rn(__uint_as_float(hi[j + 3]), b1.w);
            }
            if (un.kv == 0) {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float c = cs[16 * rnd + j], sv = sn[16 * rnd + j];
                const float y0 = ylo[j], y1 = yhi[j];
                ylo[j] = __fmaf_rn(y0, c, -__fmul_rn(y1, sv));
                yhi[j] = __fmaf_rn(y0, sv, __fmul_rn(y1, c));
              }
            }
#pragma unroll
            for (int j = 0; j < 16; j += 8) {
              const uint4 v0 = make_uint4(pack_bf16x2(ylo[j], ylo[j + 1]), pack_bf16x2(ylo[j + 2], ylo[j + 3]),
                                          pack_bf16x2(ylo[j + 4], ylo[j + 5]), pack_bf16x2(ylo[j + 6], ylo[j + 7]));
              const uint4 v1 = make_uint4(pack_bf16x2(yhi[j], yhi[j + 1]), pack_bf16x2(yhi[j + 2], yhi[j + 3]),
                                          pack_bf16x2(yhi[j + 4], yhi[j + 5]), pack_bf16x2(yhi[j + 6], yhi[j + 7]));
              st_global_stream(out + 16 * rnd + j, v0, st_pol);
              st_global_stream(out + 64 + 16 * rnd + j, v1, st_pol);
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kTmemCols)
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

size_t smem_bytes(int n_slots, int n_wst) {
  const size_t bars = (3 * n_slots + 2 * n_wst + 5) * 8 + 16;
  return 1024 + static_cast<size_t>(n_slots) * kSlotBytes + static_cast<size_t>(n_wst) * kWStageBytes + bars;
}

// Belady schedule of source-tile loads over the use sequence (l, j), l-major.
void build_plan(const kvx_ctx* c, int n_slots, TcPlan* plan) {
  const int Lt = c->Lt, k = c->k, n_uses = Lt * k;
  std::vector<int> src(n_uses), next_use(n_uses);
  for (int u = 0; u < n_uses; ++u) src[u] = c->sel[u];
  std::vector<int> seen(c->Ls, INT_MAX);
  for (int u = n_uses - 1; u >= 0; --u) {
    next_use[u] = seen[src[u]];
    seen[src[u]] = u;
  }
  plan->n_slots = n_slots;
  plan->load_layer.clear();
  plan->load_slot.clear();
  plan->load_first_use.clear();
  plan->use_slot.assign(n_uses, -1);
  plan->use_flags.assign(n_uses, 0);
  std::vector<int> slot_src(n_slots, -1), slot_next(n_slots, INT_MAX), slot_last(n_slots, -1);
  for (int u = 0; u < n_uses; ++u) {
    const int l = u / k;
    int s = -1;
    for (int i = 0; i < n_slots; ++i)
      if (slot_src[i] == src[u]) s = i;
    if (s < 0) {
      // victim: an empty slot, else the one whose next use is farthest away
      int best = -1;
      for (int i = 0; i < n_slots; ++i) {
        const int key = slot_src[i] < 0 ? INT_MAX : slot_next[i];
        if (best < 0 || key > (slot_src[best] < 0 ? INT_MAX : slot_next[best])) best = i;
        if (slot_src[i] < 0) {
          best = i;
          break;
        }
      }
      s = best;
      if (slot_src[s] >= 0) plan->use_flags[slot_last[s]] |= 2;
      plan->load_layer.push_back(src[u]);
      plan->load_slot.push_back(s);
      plan->load_first_use.push_back(l);
      slot_src[s] = src[u];
      plan->use_flags[u] |= 1;
    }
    plan->use_slot[u] = s;
    slot_next[s] = next_use[u];
    slot_last[s] = u;
  }
  for (int i = 0; i < n_slots; ++i)
    if (slot_src[i] >= 0) plan->use_flags[slot_last[i]] |= 2;
  plan->n_loads = static_cast<int>(plan->load_layer.size());
}

}  // namespace

bool tc_supported(const kvx_ctx* c, std::string* why) {
  std::string w;
  if (c->cache_dtype != KVX_BF16 || c->weight_dtype != KVX_BF16) w = "needs bf16 caches and weights";
  else if (c->d != kD) w = "needs head_dim 128";
  else if (c->head_mix != KVX_PER_HEAD) w = "needs per-head features";
  else if (c->rope_style != KVX_ROPE_HALF) w = "needs half-split RoPE pairs";
  else if (static_cast<int64_t>(c->Lt) * 2 * c->H * kD > INT_MAX) w = "too many W rows";
  if (why) *why = w;
  return w.empty();
}

kvx_status tc_prepare(kvx_ctx* c, const void* W_host) {
  // W [L_t][2][H][F][128] -> W^T [L_t][2][H][128][F] (B operand, K-major)
  const size_t F = c->F;
  const size_t blocks = static_cast<size_t>(c->Lt) * 2 * c->H;
  std::vector<uint16_t> wt(blocks * F * kD);
  const uint16_t* w = static_cast<const uint16_t*>(W_host);
  for (size_t blk = 0; blk < blocks; ++blk) {
    const uint16_t* src = w + blk * F * kD;
    uint16_t* dst = wt.data() + blk * F * kD;
    for (size_t f = 0; f < F; ++f)
      for (int n = 0; n < kD; ++n) dst[static_cast<size_t>(n) * F + f] = src[f * kD + n];
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
  // slots and W stages within the shared-memory budget
  int n_wst = 4;
  int n_slots = std::min<int>(kMaxSlots, c->k + 2);
  while (n_slots > 1 && smem_bytes(n_slots, n_wst) > kSmemLimit) --n_slots;
  while (n_wst < kMaxWStages && smem_bytes(n_slots, n_wst + 1) <= kSmemLimit) ++n_wst;
  build_plan(c, n_slots, &c->plan);
  c->plan.n_wst = n_wst;
  const TcPlan& p = c->plan;
  std::vector<int32_t> tab;
  tab.insert(tab.end(), p.load_layer.begin(), p.load_layer.end());
  tab.insert(tab.end(), p.load_slot.begin(), p.load_slot.end());
  tab.insert(tab.end(), p.load_first_use.begin(), p.load_first_use.end());
  tab.insert(tab.end(), p.use_slot.begin(), p.use_slot.end());
  tab.insert(tab.end(), p.use_flags.begin(), p.use_flags.end());
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
  // source maps: dims (d, T, H, B, L_s), strides in bytes for dims 1..4
  const cuuint64_t sdims[5] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(a.T),
                               static_cast<cuuint64_t>(c->H), static_cast<cuuint64_t>(a.B),
                               static_cast<cuuint64_t>(c->Ls)};
  const cuuint64_t sstr[4] = {static_cast<cuuint64_t>(a.ss[3]) * 2, static_cast<cuuint64_t>(a.ss[2]) * 2,
                              static_cast<cuuint64_t>(a.ss[1]) * 2, static_cast<cuuint64_t>(a.ss[0]) * 2};
  const cuuint32_t sbox[5] = {64, kTileM, 1, 1, 1};
  const cuuint32_t ones[5] = {1, 1, 1, 1, 1};
  for (int kv = 0; kv < 2; ++kv) {
    CUresult r = encode(kv ? &P.tm_v : &P.tm_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                        const_cast<void*>(kv ? a.src_v : a.src_k), sdims, sstr, sbox, ones,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      set_error("kvx_map: source tensor map rejected (strides or sizes)");
      return KVX_ERR_UNSUPPORTED;
    }
  }
  const cuuint64_t wdims[2] = {static_cast<cuuint64_t>(c->F), static_cast<cuuint64_t>(c->Lt) * 2 * c->H * kD};
  const cuuint64_t wstr[1] = {static_cast<cuuint64_t>(c->F) * 2};
  const cuuint32_t wbox[2] = {64, 128};
  CUresult r = encode(&P.tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->d_Wt, wdims, wstr, wbox, ones,
                      CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("kvx_map: weight tensor map rejected");
    return KVX_ERR_CUDA;
  }
  const TcPlan& p = c->plan;
  const int n_uses = c->Lt * c->k;
  P.a = a;
  P.load_layer = c->d_plan;
  P.load_slot = c->d_plan + p.n_loads;
  P.load_first = c->d_plan + 2 * p.n_loads;
  P.use_slot = c->d_plan + 3 * p.n_loads;
  P.use_flags = c->d_plan + 3 * p.n_loads + n_uses;
  P.bias = c->d_b;
  P.status = c->d_status;
  P.Lt = c->Lt;
  P.H = c->H;
  P.k = c->k;
  P.n_slots = p.n_slots;
  P.n_wst = p.n_wst;
  P.n_loads = p.n_loads;
  P.tiles_per_seq = (a.T + kTileM - 1) / kTileM;
  const int64_t units = static_cast<int64_t>(a.B) * P.tiles_per_seq * c->H * 2;
  if (units > INT_MAX) {
    set_error("kvx_map: too many work units");
    return KVX_ERR_UNSUPPORTED;
  }
  P.n_units = static_cast<int>(units);
  P.same_theta = c->theta_s == c->theta_t;
  P.rope = c->rope;
  const size_t smem = smem_bytes(P.n_slots, P.n_wst);
  cudaError_t e = cudaFuncSetAttribute(tc_map_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: smem attribute: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  const int grid = static_cast<int>(std::min<int64_t>(units, c->sm_count));
  tc_map_kernel<<<grid, kThreads, smem, stream>>>(P);
  e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error(std::string("kvx_map: tensor-core launch: ") + cudaGetErrorString(e));
    return KVX_ERR_CUDA;
  }
  return KVX_OK;
}

}  // namespace kvx
