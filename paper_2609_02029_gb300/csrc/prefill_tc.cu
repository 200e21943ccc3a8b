// prefill_tc.cu -- window-limited causal prefill on the 5th-generation tensor
// cores (tcgen05 + TMEM + TMA) (HeadWiseKV Sec. 3.2, Eq. conditional-attention-
// weight and Eq. conditional-attention for every prompt position; Sec. 3.3:
// each KV head reads only its own ring).
//
// Query p in [t0, t0+n) of query head q attends to KV head q/G at positions
// [max(0, p-W+1), p]: positions < t0 from the head's ring, >= t0 from the
// chunk's own K/V. The ring is walked in slot order (slot j holds the unique
// retained position congruent to j mod cap), so wrap needs no special case;
// each key column carries its position and the window/causal mask is applied
// per element on the tiles that need it. Tiles no row of the block can see are
// never loaded, so a short-window head does window-sized work.
//
// Query tile = 128 rows: 128/G positions x the G query heads of one KV head (the
// GQA group shares every K/V tile). A CTA takes QT adjacent query tiles of the
// same KV head and streams the union of their key tiles once, so every K/V tile
// brought into shared memory feeds QT x 128 rows. Warp roles:
//   warp 0      TMA producer: Q once, then K tiles into a KST-deep ring and
//               V tiles into a VST-deep ring (K runs ahead of V); with one query
//               tile per CTA the V tiles come from a producer warp of their own
//               (after the PV issuer), as one thread's copies cannot feed it
//   warp 1      QK^T issuer (one thread): per key tile, S_t = Q_t K^T for each
//               query tile t into its TMEM tile (128 x BN fp32, SBUF-buffered)
//   warps 2+    softmax, one warpgroup per query tile: thread r owns TMEM lane
//               r = query row r, so the row max and sum are thread-local; the S
//               row is read in 64-column chunks (row max, then weights, sum and
//               P); P goes back to TMEM as bf16 pairs (with PS over the first half
//               of its own S columns) and is the tensor-memory A operand of the PV
//               mma; O is rescaled in TMEM only when a row's running max grows by
//               more than 2^8 (the final O / l uses the same reference, so the
//               result is exact)
//   last warp   PV issuer (one thread): O_t += P_t V per key tile (128 x D fp32)
// Two issuing threads keep the tensor core fed while one of them waits on a
// barrier (a wait after an mma batch drains that thread's short mma queue). With
// P over one S buffer a tile's next QK^T waits for its PV, so the QT tiles of a CTA
// overlap each other's softmax and products; without PS (SBUF buffers, P apart) a
// tile's next QK^T only waits until its softmax has read S.
// All waits are bounded; a thread that gives up stops waiting and issuing but
// keeps walking the tile sequence, so every role reaches the TMEM release.
#include "hwkv_internal.cuh"

namespace hwkv {

namespace {

// D head_dim; BN keys per tile; KST / VST K and V tile buffers; QT query tiles per
// CTA; SBUF S buffers per query tile; CTAS resident CTAs per SM; PS P written over
// its S columns; F16 q, K and V (and P) in fp16 instead of bf16 (staged 8-bit cache).
template <int D, int BN, int KST, int VST, int QT, int SBUF, int CTAS, bool PS, bool F16>
struct TcCfg {
  static constexpr int kSoftmaxWarps = 4 * QT;      // one warpgroup per query tile
  // One thread's TMA tile copies reach ~45 B/clk into an SM, two threads' ~72. With
  // one query tile per CTA a key tile's K and V (4 d B per key) feed half the rows
  // they feed with two, so V tiles get a producer warp of their own.
  static constexpr bool kSplitV = QT == 1;
  // warp 0 TMA producer (K only with kSplitV), warp 1 QK^T issuer, warps 2 .. 2 + 4 QT - 1
  // softmax, warp 2 + 4 QT PV issuer, then (kSplitV) the V producer
  static constexpr int kVWarp = 3 + kSoftmaxWarps;
  static constexpr int kThreads = 96 + 32 * kSoftmaxWarps + (kSplitV ? 32 : 0);
  static_assert(BN % 32 == 0 && D % 32 == 0, "TMEM loads of 32 columns");
  static constexpr int kSlabs = D / 64;
  static constexpr int kQSlab = 128 * 128;             // 128 rows x 128 B
  static constexpr int kQTile = kSlabs * kQSlab;       // one query tile
  static constexpr int kQBytes = QT * kQTile;
  static constexpr int kKVSlab = BN * 128;             // BN rows x 128 B
  static constexpr int kTileBytes = kSlabs * kKVSlab;  // one K (or V) tile
  // TMEM columns: S of query tile t, buffer sb at kColS + (t SBUF + sb) BN; O of
  // tile t at kColO + t D; P of tile t (bf16 pairs, BN / 2 columns) at kColO + QT D +
  // t BN / 2, or with PS over the first half of the S buffer it was computed from
  static_assert(PS || BN == 64, "without P over S the S row is held in registers whole");
  static constexpr int kColS = 0;
  static constexpr int kColO = QT * SBUF * BN;
  // P-written and PV-done barriers: with PS one per S buffer (P lives in that buffer;
  // a softmax warp may run a key tile ahead of the PV issuer, so a per-tile barrier
  // could complete two phases before it is waited on), else one per query tile
  static constexpr int kPBars = PS ? QT * SBUF : QT;
  // With P over 128-key S tiles the softmax writes P in two 64-key chunks, the chunk it
  // still holds in registers first; a barrier on that half lets the PV product over
  // its 64 keys start while the softmax works on the other chunk
  static constexpr bool kHalfP = PS && BN == 128;
  static constexpr int kNumBars = 2 * KST + 2 * VST + 2 * QT * SBUF + 3 * kPBars + 4;
  static constexpr int kBarBytes = 512;
  static_assert(8 * kNumBars + 4 <= kBarBytes, "barriers and the TMEM address slot");
  // the dynamic shared memory window starts 1024-aligned (the kernel checks it)
  static constexpr int kSmem = kQBytes + (KST + VST) * kTileBytes + kBarBytes;
  static_assert(kSmem * CTAS <= 232448 - 1024 * (CTAS - 1), "shared memory per SM");
  static constexpr int kTmemNeed = PS ? kColO + QT * D : kColO + QT * D + QT * BN / 2;
  // P of key chunk ch (64 keys = 32 columns) relative to col_p: chunk 0 first; with
  // PS and two chunks the last chunk's P goes over the second half of its own S
  // columns (already in registers when its P is written), every other chunk's P
  // over the first half of chunk 0's S columns
  __device__ static constexpr uint32_t p_chunk_col(int ch) {
    return (PS && BN == 128 && ch == 1) ? 96u : (uint32_t)(ch * 32);
  }
  // first P column of query tile t for key tile j
  __device__ static constexpr uint32_t col_p(int t, uint32_t j) {
    return PS ? (uint32_t)(kColS + (t * SBUF + (int)(j % SBUF)) * BN)
              : (uint32_t)(kColO + QT * D + t * (BN / 2));
  }
  // P-written / PV-done barrier of query tile t for key tile j, and its phase parity
  __device__ static constexpr int p_bar(int t, uint32_t j) { return PS ? t * SBUF + (int)(j % SBUF) : t; }
  __device__ static constexpr uint32_t p_parity(uint32_t j) { return PS ? (j / SBUF) & 1u : j & 1u; }
  static constexpr uint32_t kTmemCols = kTmemNeed <= 128 ? 128 : (kTmemNeed <= 256 ? 256 : 512);
  static_assert(kTmemNeed <= 512 && kTmemCols * CTAS <= 512,
                "TMEM: S buffers, O and P of every query tile of every resident CTA");
};

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int32_t x,
                                            int32_t y, int32_t z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

// The key tiles one query block needs, in order: the sink slots (all read by
// every row), then tiles of the window region (slots S .. cap-1, positions >= S,
// position p in slot S + (p - S) mod Wr) whose newest held position reaches the
// block's lowest visible key, then chunk tiles up to the block's last row (from
// the chunk's start while it still holds sink positions). A ring tile's j0 is its
// first ring slot. Every role walks the same sequence. Without sinks (S = 0) the
// window region is the whole ring.
template <int BN>
struct KeySeq {
  int32_t t0, n, W, S, Wr, n_sink, tw, n_win, r0, lo_need, c_first, n_chunk_tiles;
  int32_t n_sink_tiles, n_win_tiles;
  bool win_needed;
  int32_t sink_cur, win_cur, chunk_cur;

  // positions, slots and counts are below 2^30 (the host rejects longer histories)
  __device__ void init(const PrefillUnit& u, int32_t t0_, int32_t n_, int32_t p0, int32_t p_last) {
    t0 = t0_;
    n = n_;
    W = (int32_t)u.window;
    S = (int32_t)u.sink;
    Wr = (int32_t)(u.cap - u.sink);
    n_sink = t0 < S ? t0 : S;
    tw = t0 > S ? t0 - S : 0;            // history tokens in the window region
    n_win = tw < Wr ? tw : Wr;
    r0 = tw % Wr;
    lo_need = W == 0 ? 0 : (p0 - W + 1 > 0 ? p0 - W + 1 : 0);
    n_sink_tiles = (n_sink + BN - 1) / BN;
    n_win_tiles = (n_win + BN - 1) / BN;
    // chunk keys below S are sinks, read by every row
    const int32_t c_lo = t0 < S ? 0 : (t0 > lo_need ? t0 : lo_need) - t0;
    c_first = (c_lo / BN) * BN;
    const int32_t c_hi = p_last - t0;
    n_chunk_tiles = c_hi >= c_first ? (c_hi - c_first) / BN + 1 : 0;
    win_needed = n_win > 0 && (W == 0 || p0 - W + 1 < t0);
    sink_cur = 0;
    win_cur = next_win(0);
    chunk_cur = 0;
  }
  // position held by window-region slot j (0-based within the region)
  __device__ int32_t slot_pos(int32_t j) const {
    if (tw <= Wr) return S + j;
    return S + (j < r0 ? tw - r0 + j : tw - r0 - Wr + j);
  }
  // largest position held in window-region slots [j0, j1] (j1 < n_win)
  __device__ int32_t tile_max_pos(int32_t j0, int32_t j1) const {
    if (tw > Wr && j0 < r0 && r0 <= j1) return slot_pos(r0 - 1);
    return slot_pos(j1);
  }
  __device__ bool win_tile_needed(int32_t jt) const {
    if (!win_needed) return false;
    if (W == 0) return true;
    const int32_t j0 = jt * BN;
    const int32_t j1 = (j0 + BN < n_win ? j0 + BN : n_win) - 1;
    return tile_max_pos(j0, j1) >= lo_need;
  }
  __device__ int32_t next_win(int32_t jt) const {
    for (; jt < n_win_tiles; ++jt)
      if (win_tile_needed(jt)) return jt;
    return -1;
  }
  // hist: 0 = chunk tile, 1 = window-region tile, 2 = sink tile
  __device__ bool next(int& hist, int32_t& j0) {
    if (sink_cur < n_sink_tiles) {
      hist = 2;
      j0 = sink_cur * BN;
      ++sink_cur;
      return true;
    }
    if (win_cur >= 0) {
      hist = 1;
      j0 = S + win_cur * BN;
      win_cur = next_win(win_cur + 1);
      return true;
    }
    if (chunk_cur < n_chunk_tiles) {
      hist = 0;
      j0 = c_first + chunk_cur * BN;
      ++chunk_cur;
      return true;
    }
    return false;
  }
};

// max of three floats in one instruction
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, int* err,
                                              bool& aborted) {
  if (aborted) return false;
  if (!mbar_wait_bounded(bar, parity, err)) aborted = true;
  return !aborted;
}

// one lane of the warp waits, the warp then proceeds together; the abort flag
// is shared by the warp so every lane takes the same path
__device__ __forceinline__ bool warp_wait_or_abort(uint64_t* bar, uint32_t parity, int* err,
                                                   bool& aborted) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = wait_or_abort(bar, parity, err, aborted) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  aborted = ok == 0;
  return ok != 0;
}

}  // namespace

template <int D, int BN, int KST, int VST, int QT, int SBUF, int CTAS, bool PS, bool F16>
__global__ void __launch_bounds__(TcCfg<D, BN, KST, VST, QT, SBUF, CTAS, PS, F16>::kThreads, CTAS)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap q_map,
                      const __grid_constant__ CUtensorMap ck_map,
                      const __grid_constant__ CUtensorMap cv_map,
                      const __grid_constant__ CUtensorMap ring_map, const PrefillParams p) {
  using C = TcCfg<D, BN, KST, VST, QT, SBUF, CTAS, PS, F16>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // the 128-byte swizzle atoms need a 1024-aligned base; stop before any copy if
  // the launch ever provides less
  if ((smem_u32(smem_raw) & 1023u) != 0u) {
    if (threadIdx.x == 0) atomicOr(p.err, kErrBadIndex);
    return;
  }
  uint8_t* smem = smem_raw;
  // K and V tiles live in separate buffers, released separately: a K buffer as soon
  // as its QK^T is done, a V buffer when its PV is done, so the next K tiles load
  // while this tile's softmax and PV run
  uint8_t* sQ = smem;                                 // [QT] query tiles
  uint8_t* sK = smem + C::kQBytes;                   // [KST] K tiles
  uint8_t* sV = sK + KST * C::kTileBytes;            // [VST] V tiles
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + VST * C::kTileBytes);
  uint64_t* k_full = bars;                    // [KST] K tile landed
  uint64_t* k_empty = k_full + KST;           // [KST] QK^T of that tile done
  uint64_t* v_full = k_empty + KST;           // [VST] V tile landed
  uint64_t* v_empty = v_full + VST;           // [VST] PV of that tile done
  uint64_t* s_full = v_empty + VST;           // [QT][SBUF] S tile computed
  uint64_t* s_free = s_full + QT * SBUF;      // [QT][SBUF] S tile read by the softmax warps
  uint64_t* p_full = s_free + QT * SBUF;      // [kPBars] P written (and O rescaled)
  uint64_t* pv_done = p_full + C::kPBars;     // [kPBars] PV mma done
  uint64_t* q_full = pv_done + C::kPBars;
  uint64_t* o_full = q_full + 1;
  uint64_t* drain = o_full + 1;               // [2] each issuer's mmas done
  uint64_t* p_half = drain + 2;               // [kPBars] first P chunk written (kHalfP)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(p_half + C::kPBars);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.group;
  const int QP = 128 / G;           // query positions per tile
  const int rows_valid = QP * G;    // rows that carry a (position, head)
  const int n_qblocks = (int)((p.n + QP - 1) / QP);
  const int n_ctas = (n_qblocks + QT - 1) / QT;
  const int qb0 = (n_ctas - 1 - (int)blockIdx.x) * QT;  // first query tile; longest rows first
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  const PrefillUnit& u = p.u[h];
  const int32_t t0 = (int32_t)p.t0;                      // positions are below 2^30
  const int32_t n_chunk = (int32_t)p.n;
  const int32_t p0 = t0 + qb0 * QP;                      // lowest position of the CTA
  const int32_t p_last = min(p0 + QT * QP, t0 + n_chunk) - 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < KST; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < VST; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int i = 0; i < QT * SBUF; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 4);  // one arrival per warp of the tile's warpgroup
    }
    for (int i = 0; i < C::kPBars; ++i) {
      mbar_init(&p_full[i], 4);  // one arrival per warp of the tile's warpgroup
      mbar_init(&p_half[i], 4);
      mbar_init(&pv_done[i], 1);
    }
    mbar_init(q_full, 1);
    mbar_init(o_full, 1);
    mbar_init(&drain[0], 1);
    mbar_init(&drain[1], 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // the union of the key tiles the CTA's query tiles need (a tile one of them
  // does not see is masked out of its rows)
  KeySeq<BN> seq;
  seq.init(u, t0, n_chunk, p0, p_last);
  bool aborted = false;

  if (C::kSplitV && (warp == 0 || warp == C::kVWarp)) {
    // ------------------------------------------------- K and V producers (kSplitV)
    // warp 0 copies Q and the K tiles, warp kVWarp the V tiles, each walking the key
    // sequence into its own ring
    if (lane == 0) {
      const bool is_k = warp == 0;
      if (is_k) {
        prefetch_tensormap(&q_map);
        prefetch_tensormap(&ck_map);
      }
      prefetch_tensormap(&cv_map);
      prefetch_tensormap(&ring_map);
      if (is_k) {
        // the query tile's box is copied whole, so the byte count is fixed
        mbar_arrive_expect_tx(q_full, (uint32_t)(QT * C::kSlabs * rows_valid * 128));
#pragma unroll
        for (int t = 0; t < QT; ++t) {
          const int32_t qrow = (int32_t)((int64_t)b * p.n + (int64_t)(qb0 + t) * QP);
#pragma unroll
          for (int sl = 0; sl < C::kSlabs; ++sl)
            tma_load_3d(sQ + t * C::kQTile + sl * C::kQSlab, &q_map, sl * 64, h * G, qrow, q_full);
        }
      }
      const int nbuf = is_k ? KST : VST;
      uint64_t* full = is_k ? k_full : v_full;
      uint64_t* empty = is_k ? k_empty : v_empty;
      uint8_t* buf = is_k ? sK : sV;
      const CUtensorMap* cmap = is_k ? &ck_map : &cv_map;
      const int64_t row0 = (is_k ? u.k_row0 : u.v_row0) + (int64_t)(p.row0 + b) * u.stride;
      uint32_t it = 0;
      int hist;
      int32_t j0;
      while (seq.next(hist, j0)) {
        const int s = it % nbuf;
        if (wait_or_abort(&empty[s], ((it / nbuf) & 1u) ^ 1u, p.err, aborted)) {
          uint8_t* d = buf + s * C::kTileBytes;
          mbar_arrive_expect_tx(&full[s], C::kTileBytes);
#pragma unroll
          for (int sl = 0; sl < C::kSlabs; ++sl) {
#pragma unroll
            for (int hf = 0; hf < BN / 64; ++hf) {
              const uint32_t off = sl * C::kKVSlab + hf * 64 * 128;
              if (hist)
                tma_load_2d(d + off, &ring_map, sl * 64, (int32_t)(row0 + j0 + hf * 64), &full[s]);
              else
                tma_load_3d(d + off, cmap, sl * 64, h, (int32_t)((int64_t)b * p.n + j0 + hf * 64),
                            &full[s]);
            }
          }
        }
        ++it;
      }
      // every copy this thread issued has landed before shared memory can go away
      bool late = false;
      for (uint32_t j = it > (uint32_t)nbuf ? it - nbuf : 0u; j < it; ++j)
        wait_or_abort(&full[j % nbuf], (j / nbuf) & 1u, p.err, late);
    }
  } else if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      prefetch_tensormap(&q_map);
      prefetch_tensormap(&ck_map);
      prefetch_tensormap(&cv_map);
      prefetch_tensormap(&ring_map);
      // every tile's box is copied whole (rows past the chunk's end read zeros or
      // the next row's queries and are masked), so the byte count is fixed
      mbar_arrive_expect_tx(q_full, (uint32_t)(QT * C::kSlabs * rows_valid * 128));
#pragma unroll
      for (int t = 0; t < QT; ++t) {
        const int32_t qrow = (int32_t)((int64_t)b * p.n + (int64_t)(qb0 + t) * QP);
#pragma unroll
        for (int sl = 0; sl < C::kSlabs; ++sl)
          tma_load_3d(sQ + t * C::kQTile + sl * C::kQSlab, &q_map, sl * 64, h * G, qrow, q_full);
      }
      const int64_t krow0 = u.k_row0 + (int64_t)(p.row0 + b) * u.stride;
      const int64_t vrow0 = u.v_row0 + (int64_t)(p.row0 + b) * u.stride;
      // two walks of the same key sequence: K tiles run one tile ahead of V tiles
      KeySeq<BN> seq_v = seq;
      uint32_t it_k = 0, it_v = 0;
      auto issue = [&](KeySeq<BN>& sq, uint32_t& it, uint64_t* full, uint64_t* empty,
                       uint8_t* buf, int64_t row0, const CUtensorMap* cmap, int nbuf) -> bool {
        int hist;
        int32_t j0;
        if (!sq.next(hist, j0)) return false;
        const int s = it % nbuf;
        const uint32_t ph = (it / nbuf) & 1u;
        if (wait_or_abort(&empty[s], ph ^ 1u, p.err, aborted)) {
          uint8_t* d = buf + s * C::kTileBytes;
          mbar_arrive_expect_tx(&full[s], C::kTileBytes);
#pragma unroll
          for (int sl = 0; sl < C::kSlabs; ++sl) {
#pragma unroll
            for (int hf = 0; hf < BN / 64; ++hf) {
              const uint32_t off = sl * C::kKVSlab + hf * 64 * 128;
              if (hist)
                tma_load_2d(d + off, &ring_map, sl * 64, (int32_t)(row0 + j0 + hf * 64), &full[s]);
              else
                tma_load_3d(d + off, cmap, sl * 64, h, (int32_t)((int64_t)b * p.n + j0 + hf * 64),
                            &full[s]);
            }
          }
        }
        ++it;
        return true;
      };
      // issue order K_{j+L} before V_j with L = KST - VST + 1: the QK^T that frees
      // K_{j+L}'s slot and the PV that frees V_j's slot depend only on copies issued
      // before them, and with the deeper K ring a K copy is not held back behind a
      // V slot that frees later than its own
      constexpr int kLead = KST - VST + 1;
      int lead = 0;  // K tiles issued minus V tiles issued
      bool more_k = true;
      while (true) {
        while (more_k && lead <= kLead) {
          more_k = issue(seq, it_k, k_full, k_empty, sK, krow0, &ck_map, KST);
          if (more_k) ++lead;
        }
        if (!issue(seq_v, it_v, v_full, v_empty, sV, vrow0, &cv_map, VST)) break;
        --lead;
      }
      // every issued copy has landed before shared memory can go away
      bool late = false;
      for (uint32_t j = it_k > (uint32_t)KST ? it_k - KST : 0u; j < it_k; ++j)
        wait_or_abort(&k_full[j % KST], (j / KST) & 1u, p.err, late);
      for (uint32_t j = it_v > (uint32_t)VST ? it_v - VST : 0u; j < it_v; ++j)
        wait_or_abort(&v_full[j % VST], (j / VST) & 1u, p.err, late);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------- QK^T issuer
    // The QK^T and PV products are issued by two threads: a thread that waits on
    // a barrier stops feeding the tensor core, and a 128 x 64 x 16 or 128 x 128 x 16
    // mma is too short to cover that wait from one thread's queue alone.
    if (lane == 0) {
      constexpr uint32_t idesc_qk = F16 ? idesc_f16_f32(128, BN, false) : idesc_bf16_f32(128, BN, false);
      const uint32_t q_base = smem_u32(sQ);
      wait_or_abort(q_full, 0, p.err, aborted);
      uint32_t j = 0;
      int hist;
      int32_t j0;
      while (seq.next(hist, j0)) {
        const int s = j % KST;
        const int sb = j % SBUF;
        bool ok = wait_or_abort(&k_full[s], (j / KST) & 1u, p.err, aborted);
        const uint32_t k_base = smem_u32(sK + s * C::kTileBytes);
#pragma unroll
        for (int t = 0; t < QT; ++t) {
          // the S buffer is free once the softmax has read it or, with P written
          // over S, once the PV product of the previous key tile has read P
          if constexpr (PS) {
            if (j >= SBUF) ok = ok && wait_or_abort(&pv_done[C::p_bar(t, j)], C::p_parity(j - SBUF), p.err, aborted);
          } else {
            ok = ok && wait_or_abort(&s_free[t * SBUF + sb], ((j / SBUF) & 1u) ^ 1u, p.err, aborted);
          }
          if (ok) {
            tc_fence_after();
            const uint32_t qt_base = q_base + t * C::kQTile;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint64_t a = smem_desc_sw128(qt_base + (kk >> 2) * C::kQSlab + (kk & 3) * 32, 16, 1024);
              const uint64_t bd = smem_desc_sw128(k_base + (kk >> 2) * C::kKVSlab + (kk & 3) * 32, 16, 1024);
              umma_bf16(tmem + C::kColS + (t * SBUF + sb) * BN, a, bd, idesc_qk, kk > 0 ? 1u : 0u);
            }
            umma_commit(&s_full[t * SBUF + sb]);
          }
        }
        if (ok) umma_commit(&k_empty[s]);  // the K tile is free once every QK^T has read it
        ++j;
      }
      // every mma this thread issued has finished before TMEM is released
      umma_commit(&drain[0]);
      bool late = false;
      wait_or_abort(&drain[0], 0, p.err, late);
    }
  } else if (warp == 2 + C::kSoftmaxWarps) {
    // ------------------------------------------------------------- PV issuer
    if (lane == 0) {
      constexpr uint32_t idesc_pv = F16 ? idesc_f16_f32(128, D, true) : idesc_bf16_f32(128, D, true);
      uint32_t j = 0;
      int hist;
      int32_t j0;
      while (seq.next(hist, j0)) {
        bool ok = wait_or_abort(&v_full[j % VST], (j / VST) & 1u, p.err, aborted);
        const uint32_t v_base = smem_u32(sV + (j % VST) * C::kTileBytes);
#pragma unroll
        for (int t = 0; t < QT; ++t) {
          // 16 keys = 8 packed P columns; with kHalfP keys 64 .. 127 (the chunk the
          // softmax writes first) go as soon as their P is written, then keys 0 .. 63
          auto pv_keys = [&](int kk0, int kk1, bool first) {
            tc_fence_after();
#pragma unroll
            for (int kk = kk0; kk < kk1; ++kk) {
              const uint64_t bd = smem_desc_sw128(v_base + kk * 2048, C::kKVSlab, 1024);
              umma_bf16_tmem_a(tmem + C::kColO + t * D, tmem + C::col_p(t, j) + C::p_chunk_col(kk / 4) + (kk % 4) * 8, bd,
                               idesc_pv, (j > 0 || !first || kk > kk0) ? 1u : 0u);
            }
          };
          if constexpr (C::kHalfP) {
            ok = ok && wait_or_abort(&p_half[C::p_bar(t, j)], C::p_parity(j), p.err, aborted);
            if (ok) pv_keys(4, 8, true);
            ok = ok && wait_or_abort(&p_full[C::p_bar(t, j)], C::p_parity(j), p.err, aborted);
            if (ok) pv_keys(0, 4, false);
          } else {
            ok = ok && wait_or_abort(&p_full[C::p_bar(t, j)], C::p_parity(j), p.err, aborted);
            if (ok) pv_keys(0, BN / 16, true);
          }
          if (ok) umma_commit(&pv_done[C::p_bar(t, j)]);
        }
        if (ok) umma_commit(&v_empty[j % VST]);  // every query tile's PV has read it
        ++j;
      }
      if (!aborted) umma_commit(o_full);
      umma_commit(&drain[1]);
      bool late = false;
      wait_or_abort(&drain[1], 0, p.err, late);
    }
  } else {
    // ---------------------------------------------------------------- softmax
    const int quarter = warp & 3;         // TMEM lanes this warp may access
    const int tq = (warp - 2) >> 2;       // this warpgroup's query tile
    const int r = quarter * 32 + lane;
    const int32_t pr = t0 + (qb0 + tq) * QP + r / G;
    const bool row_ok = r < rows_valid && pr <= p_last;
    const uint32_t colS = C::kColS + tq * SBUF * BN;  // this tile's S buffers
    const uint32_t colO = C::kColO + tq * D;
    const int qh = h * G + r % G;
    const int32_t W = seq.W;
    const int32_t lo_r = W == 0 ? 0 : (pr - W + 1 > 0 ? pr - W + 1 : 0);  // first visible key
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16);
    const float c = p.scale_log2;
    float m_used = -INFINITY, l = 0.f;  // running max (log2 units) and sum of weights
    uint32_t j = 0;
    int hist;
    int32_t j0;
    auto clampi = [](int32_t v) -> int { return v < -1 ? -1 : (v > BN + 1 ? BN + 1 : v); };
    while (seq.next(hist, j0)) {
      const int sb = j % SBUF;
      // columns e of this tile visible to row pr: [a0, b0) U [a1, b1)
      int a0 = 0, b0 = 0, a1 = 0, b1 = 0;
      if (row_ok) {
        if (hist == 0) {  // chunk keys at positions t0 + j0 + e, held while j0 + e < n
          const int32_t hi = min(pr - t0 - j0, n_chunk - 1 - j0);  // causal, held
          a0 = clampi(lo_r - t0 - j0);
          b0 = clampi(hi + 1);
          b1 = clampi(min(seq.S - t0 - j0, hi + 1));  // chunk keys that are sinks
        } else if (hist == 2) {  // sink slots: slot j holds position j, always visible
          b0 = clampi(seq.n_sink - j0);
        } else {
          // window region, slots relative to its start: position S + v in slot
          // S + (v mod Wr) for the region's v-th held token
          const int32_t jw = j0 - seq.S, lo_v = lo_r - seq.S;
          if (seq.tw <= seq.Wr) {  // not yet wrapped
            a0 = clampi(lo_v - jw);
            b0 = clampi(seq.n_win - jw);
          } else {  // wrapped: slots < r0 hold the newest run, slots >= r0 the older one
            const int32_t A = lo_v - seq.tw + seq.r0;  // first visible slot of the newest run
            a0 = clampi(A - jw);
            b0 = clampi(seq.r0 - jw);
            a1 = clampi(A + seq.Wr - jw);
            b1 = clampi(seq.Wr - jw);
          }
        }
      }
      // A row that carries no (position, head) (the tile's last 128 mod G rows, or
      // rows past the chunk) counts as fully visible: its output is never stored and
      // it never rescales O, so it does not hold its warp on the masked path.
      const bool full_vis = !row_ok || (a0 <= 0 && b0 >= BN) || (a1 <= 0 && b1 >= BN);
      const bool warp_full = __all_sync(0xffffffffu, full_vis);  // warp-uniform fast path
      if (warp_wait_or_abort(&s_full[tq * SBUF + sb], (j / SBUF) & 1u, p.err, aborted)) tc_fence_after();
      // The S row in chunks of 64 columns: pass 1 takes the row max, pass 2 the
      // weights, the row sum and P. With one chunk the registers carry over; with
      // more the chunk is read from TMEM again (P over S overwrites only columns
      // of chunks already read).
      constexpr int kChunks = BN / 64;
      uint32_t sv[64];
      auto load_chunk = [&](int ch) {
        tmem_ld32(t_lane + colS + sb * BN + ch * 64, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
        tmem_ld32(t_lane + colS + sb * BN + ch * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
        tmem_ld_wait();
        if (!warp_full) {  // masked logits -> -inf (weight 0)
#pragma unroll
          for (int e = 0; e < 64; ++e) {
            const int col = ch * 64 + e;
            const bool vis = full_vis || (col >= a0 && col < b0) || (col >= a1 && col < b1);
            if (!vis) sv[e] = __float_as_uint(-INFINITY);
          }
        }
      };
      // row max of the visible logits (raw; scale > 0 so max(z) c = max(z c))
      float mx;
      {
        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int ch = 0; ch < kChunks; ++ch) {
          load_chunk(ch);
#pragma unroll
          for (int e = 0; e < 64; e += 8)
#pragma unroll
            for (int i = 0; i < 4; ++i)
              m4[i] = fmax3(m4[i], __uint_as_float(sv[e + i]), __uint_as_float(sv[e + 4 + i]));
        }
        mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
        mx *= c;
      }
      if constexpr (!PS) {
        // the S row is in registers: the buffer is free for the QK^T of key tile j + SBUF
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[tq * SBUF + sb]);
      }
      const float m_new = fmaxf(m_used, mx);
      const bool resc = row_ok && m_new - m_used > 8.f;  // false while both are -inf
      float alpha = 1.f;
      if (resc) {
        alpha = ex2(m_used - m_new);
        m_used = m_new;
        l *= alpha;
      }
      const float bias = m_used == -INFINITY ? 0.f : m_used;
      // O *= alpha (rare: the reference max only moves when a row's max grows by more
      // than 2^8). The PV product of the previous key tile must have added into O.
      auto rescale_o = [&]() {
        if (j >= 1 && __any_sync(0xffffffffu, resc)) {
          const uint32_t tO = t_lane + colO;
#pragma unroll
          for (int cc = 0; cc < D / 32; ++cc) {
            uint32_t rr[32];
            tmem_ld32(tO + cc * 32, rr);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) rr[e] = __float_as_uint(__uint_as_float(rr[e]) * alpha);
            tmem_st32(tO + cc * 32, rr);
          }
        }
      };
      // With P over S and one S buffer that product finished before this tile's QK^T
      // was issued; with more S buffers it is waited for when a row rescales.
      if constexpr (PS) {
        if (SBUF > 1 && j >= 1 && __any_sync(0xffffffffu, resc) &&
            warp_wait_or_abort(&pv_done[C::p_bar(tq, j - 1)], C::p_parity(j - 1), p.err, aborted))
          tc_fence_after();
        rescale_o();
      }

      // weights 2^(z c - m) (masked logits are -inf: weight 0); the exponent
      // arguments and the row sum in packed fp32 pairs; P as bf16 pairs
      float2 s2a = make_float2(0.f, 0.f), s2b = make_float2(0.f, 0.f);
      // the last chunk is still in registers: it goes first; the others are read again
#pragma unroll
      for (int cc = 0; cc < kChunks; ++cc) {
        const int ch = (cc + kChunks - 1) % kChunks;
        if (cc > 0) load_chunk(ch);
        const float2 c2 = make_float2(c, c), nb2 = make_float2(-bias, -bias);
#pragma unroll
        for (int e = 0; e < 64; e += 2) {
          const float2 y = fma2(make_float2(__uint_as_float(sv[e]), __uint_as_float(sv[e + 1])), c2, nb2);
          const float2 w = make_float2(ex2(y.x), ex2(y.y));
          if (e & 2) s2b = add2(s2b, w); else s2a = add2(s2a, w);
          // in place: index e / 2 was already read; P in the operands' type
          sv[e / 2] = F16 ? pack_f16(w.x, w.y) : pack_bf16(w.x, w.y);
        }
        if constexpr (!PS) {
          // P is single-buffered apart from S: the previous PV must have read it
          if (j >= 1 && warp_wait_or_abort(&pv_done[C::p_bar(tq, j - 1)], C::p_parity(j - 1), p.err, aborted))
            tc_fence_after();
          rescale_o();
        }
        tmem_st32(t_lane + C::col_p(tq, j) + C::p_chunk_col(ch), *reinterpret_cast<const uint32_t(*)[32]>(&sv[0]));
        if constexpr (C::kHalfP) {
          if (cc == 0) {  // this chunk's P (and any O rescale before it) is in TMEM
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_half[C::p_bar(tq, j)]);
          }
        }
      }
      tmem_st_wait();
      float s4[4] = {s2a.x, s2a.y, s2b.x, s2b.y};
      const float sum = (s4[0] + s4[1]) + (s4[2] + s4[3]);
      l += sum;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[C::p_bar(tq, j)]);  // P rows written (and O rescaled)
      ++j;
    }
    // epilogue: O / l for this row
    if (warp_wait_or_abort(o_full, 0, p.err, aborted)) tc_fence_after();
    const float inv = l > 0.f ? 1.f / l : 0.f;
    float* dst = p.out + (((int64_t)b * p.n + (pr - t0)) * p.n_q_heads + qh) * D;
#pragma unroll
    for (int cc = 0; cc < D / 32; ++cc) {
      uint32_t rr[32];
      tmem_ld32(t_lane + colO + cc * 32, rr);
      tmem_ld_wait();
      if (row_ok) {
#pragma unroll
        for (int e = 0; e < 32; e += 4)
          *reinterpret_cast<float4*>(dst + cc * 32 + e) =
              make_float4(__uint_as_float(rr[e]) * inv, __uint_as_float(rr[e + 1]) * inv,
                          __uint_as_float(rr[e + 2]) * inv, __uint_as_float(rr[e + 3]) * inv);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

template <int D, int BN, int KST, int VST, int QT, int SBUF, int CTAS, bool PS, bool F16>
static cudaError_t launch_tc(const PrefillParams& p, const CUtensorMap& qm, const CUtensorMap& km,
                             const CUtensorMap& vm, const CUtensorMap& rm, cudaStream_t s) {
  using C = TcCfg<D, BN, KST, VST, QT, SBUF, CTAS, PS, F16>;
  cudaError_t e = cudaFuncSetAttribute(prefill_tc_kernel<D, BN, KST, VST, QT, SBUF, CTAS, PS, F16>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  const int QP = 128 / p.group;
  const int64_t n_qblocks = (p.n + QP - 1) / QP;
  dim3 grid((unsigned)((n_qblocks + QT - 1) / QT), (unsigned)p.n_units, (unsigned)p.batch);
  prefill_tc_kernel<D, BN, KST, VST, QT, SBUF, CTAS, PS, F16><<<grid, C::kThreads, C::kSmem, s>>>(qm, km, vm, rm, p);
  return cudaGetLastError();
}

int prefill_tc_rows_per_tile(int group) { return (128 / group) * group; }

cudaError_t launch_prefill_tc(const PrefillParams& p, int head_dim, const CUtensorMap& q_map,
                              const CUtensorMap& ck_map, const CUtensorMap& cv_map,
                              const CUtensorMap& ring_map, cudaStream_t s, bool fp8) {
  if (p.n == 0) return cudaSuccess;
  if (fp8) {  // staged 8-bit cache: q, K and V tiles in fp16 (head_dim 128 and 256)
    switch (head_dim) {
      case 128: return launch_tc<128, 128, 3, 2, 2, 1, 1, true, true>(p, q_map, ck_map, cv_map, ring_map, s);
      case 256: return launch_tc<256, 64, 2, 3, 1, 2, 1, false, true>(p, q_map, ck_map, cv_map, ring_map, s);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (head_dim) {
    // <head_dim, keys per tile, K buffers, V buffers, query tiles, S buffers, CTAs per SM,
    //  P over S>
    case 64: return launch_tc<64, 128, 4, 4, 2, 1, 1, true, false>(p, q_map, ck_map, cv_map, ring_map, s);
    case 128: return launch_tc<128, 128, 3, 2, 2, 1, 1, true, false>(p, q_map, ck_map, cv_map, ring_map, s);
    case 256: return launch_tc<256, 64, 2, 3, 1, 2, 1, false, false>(p, q_map, ck_map, cv_map, ring_map, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hwkv
