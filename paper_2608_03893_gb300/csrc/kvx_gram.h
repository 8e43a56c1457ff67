// Centred second-moment blocks on the tensor cores (kvx_gram.cu), shared by the ridge fit
// (kvx_fit.cu) and the R^2 probe.
#pragma once

#include "kvx_internal.h"

namespace kvx {

// An operand is one (side, layer, K|V, head) of a bf16 cache, head_dim
// 128, half-split pairs: keys with their RoPE stripped (theta_s for side 0, theta_t for
// side 1), values as stored, both centred by the column means over the N = B T tokens.
struct GramCache {
  const void* k;
  const void* v;
  int64_t s[4];                     // strides (layer, batch, head, token), elements
};

struct GramSpec {
  GramCache cache[2];               // side 0: source cache, side 1: target cache
  const int32_t* pos;               // device [B][T]
  int32_t B = 0, T = 0, H = 0, Ls = 0, Lt = 0;
  RopeTables rope{};
  int32_t hf = 0;                   // strip with the HF numerics (kvx_rope_numerics)
  std::vector<int32_t> slot_side;   // host: the operands' (side, layer), one per slot
  std::vector<int32_t> slot_layer;
  double* sums = nullptr;           // device [2 sides][2 kv][L][H][128] (side 0: L_s rows,
                                    // side 1: L_t rows), zeroed by the caller; filled by
                                    // gram_sums for every slot
  double* sumsq = nullptr;          // device [n_slots][2][H] sum of squares of the centred
                                    // operand (zeroed by the caller), or NULL
  int32_t* status = nullptr;        // device status word
  int sm_count = 0;
};

// One 128 x 128 block out[i][j] = sum_n A[n][i] B[n][j] of two centred operands (slots):
// A is head h of slot a_slot, B head hb of slot b_slot (hb < 0: the same head h).
struct GramBlock {
  int32_t a_slot, b_slot, kv, h;
  float* out;                       // device, fp32 row-major
  int32_t hb = -1;
};

// Device time of the phases of one offline call (fit or probe), from CUDA events on the
// call's stream: 0 column sums, 1 operand packing, 2 tensor-core Gram blocks, 3 solve /
// score.  finish() (after the stream is synchronised) publishes the sums for
// kvx_last_phase_ms on this thread.
class PhaseTimer {
 public:
  explicit PhaseTimer(cudaStream_t s) : stream_(s) {}
  ~PhaseTimer();
  void begin(int phase);
  void end();
  void finish();

 private:
  cudaStream_t stream_;
  int open_ = -1;
  std::vector<int> phase_;
  std::vector<cudaEvent_t> ev_;
};

// A caller-provided device region that the offline calls carve their workspace from (256-
// byte aligned pieces from the front); with p == NULL they allocate stream-ordered memory.
struct Scratch {
  char* p = nullptr;
  size_t bytes = 0;
  char* take(size_t n) {
    const size_t a = (n + 255) / 256 * 256;
    if (!p || a > bytes) return nullptr;
    char* r = p;
    p += a;
    bytes -= a;
    return r;
  }
};

// Bytes gram_sums and gram_blocks take from a Scratch besides the packed operands (slot
// tables, work units, means; `n_blocks` blocks), and bytes of packed operands per token.
size_t gram_fixed_bytes(const GramSpec& spec, size_t n_blocks);
size_t gram_bytes_per_token(const GramSpec& spec);

// Column sums of every slot into spec.sums (one pass over the caches).
kvx_status gram_sums(const GramSpec& spec, cudaStream_t stream, PhaseTimer* timer, Scratch* scratch);
// Every block of the list (after gram_sums); the tokens are processed in chunks that
// keep the packed operands within `ws_budget` bytes, or, with a Scratch, within what is
// left of it.
kvx_status gram_blocks(const GramSpec& spec, const std::vector<GramBlock>& blocks, size_t ws_budget,
                       cudaStream_t stream, PhaseTimer* timer, Scratch* scratch);
}  // namespace kvx
