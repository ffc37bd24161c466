// env_hanabi.cuh -- 2-player Hanabi on the device (one thread per env).
//
// 50-card deck (5 colours x ranks 1,1,1,2,2,3,3,4,4,5), 5-card hands, 8 info and 3 life
// tokens, 20 actions (play slot 0-4, discard slot 0-4, hint colour 0-4, hint rank 1-5),
// seat 0 first.  Card type = colour*5 + rank-1.  Play is legal for an occupied slot,
// discard also needs info < 8, a hint needs info > 0 and a matching partner card; a
// successful play pays +1 (a completed 5 returns an info token), losing the last life
// zeroes the return; the game ends at 0 lives, score 25, or two turns after the draw that
// empties the deck.  The 660-bit observation (Sec. 4 Table, Hanabi; layout ours) is laid
// out section by section in obs_into.
#pragma once
#include "aht_common.cuh"

namespace aht {

struct EnvHanabi {
  static constexpr bool kTurnBased = true;
  static constexpr int kNumActions = 20;
  static constexpr int kTurnCap = 100;
  struct State {
    uint8_t deck[52];
    uint8_t hand[2][5];
    uint8_t n_hand[2];
    uint32_t know[2][5];    // possible card types, 25 bits
    uint16_t hints[2][5];   // explicit hints received: bits 0-4 colour, 5-9 rank
    uint8_t fw[5], info, lives, score;
    uint8_t disc[25], ptr, turn;
    int8_t fr;              // final-round turns left, -1 while the deck has cards
    uint8_t la_flags;       // bit0 valid, bit1 actor seat, bit2 play success, bit3 bomb
    uint8_t la_type, la_colour, la_rank, la_slot, la_card, la_hinted, la_pad;
    float ret;
  };
  static constexpr int kWords = sizeof(State) / 4;

  __device__ static uint32_t colour_bits(int c) { return 0x1Fu << (5 * c); }
  __device__ static uint32_t rank_bits(int r0) { return 0x108421u << r0; }  // rank index 0..4

  __device__ static void reset(const DevEnv&, Key key, uint32_t env, uint32_t step, State& s) {
    // canonical order: colour c, copies of ranks 1,1,1,2,2,3,3,4,4,5
    for (int c = 0; c < 5; ++c) {
      uint8_t* p = s.deck + c * 10;
      const uint8_t b = (uint8_t)(c * 5);
      p[0] = p[1] = p[2] = b;
      p[3] = p[4] = b + 1;
      p[5] = p[6] = b + 2;
      p[7] = p[8] = b + 3;
      p[9] = b + 4;
    }
    s.deck[50] = s.deck[51] = 0;
    DrawSeq r(key, env, step, kStreamReset);
    for (int i = 49; i >= 1; --i) {
      const int j = (int)uniform_int(r.next(), (uint32_t)(i + 1));
      const uint8_t t = s.deck[i];
      s.deck[i] = s.deck[j];
      s.deck[j] = t;
    }
    for (int p = 0; p < 2; ++p) {
      for (int k = 0; k < 5; ++k) {
        s.hand[p][k] = s.deck[p * 5 + k];
        s.know[p][k] = 0x1FFFFFFu;
        s.hints[p][k] = 0;
      }
      s.n_hand[p] = 5;
    }
    for (int c = 0; c < 5; ++c) s.fw[c] = 0;
    for (int t = 0; t < 25; ++t) s.disc[t] = 0;
    s.info = 8;
    s.lives = 3;
    s.score = 0;
    s.ptr = 10;
    s.turn = 0;
    s.fr = -1;
    s.la_flags = 0;
    s.la_type = s.la_colour = s.la_rank = s.la_slot = s.la_card = s.la_hinted = s.la_pad = 0;
    s.ret = 0.0f;
  }

  __device__ static int actor(const State& s) { return s.turn & 1; }

  __device__ static uint32_t legal(const State& s) {
    const int me = s.turn & 1, pa = me ^ 1;
    uint32_t m = 0;
    for (int k = 0; k < s.n_hand[me]; ++k) {
      m |= 1u << k;
      if (s.info < 8) m |= 1u << (5 + k);
    }
    if (s.info > 0) {
      for (int k = 0; k < s.n_hand[pa]; ++k) {
        const int card = s.hand[pa][k];
        m |= 1u << (10 + card / 5);
        m |= 1u << (15 + card % 5);
      }
    }
    return m;
  }

  __device__ static void remove_slot(State& s, int p, int slot) {
    const int n = s.n_hand[p];
    for (int k = slot; k < n - 1; ++k) {
      s.hand[p][k] = s.hand[p][k + 1];
      s.know[p][k] = s.know[p][k + 1];
      s.hints[p][k] = s.hints[p][k + 1];
    }
    s.hand[p][n - 1] = 0;
    s.know[p][n - 1] = 0;
    s.hints[p][n - 1] = 0;
    s.n_hand[p] = (uint8_t)(n - 1);
  }

  // Applies the acting seat's action (a0 for seat 0, a1 for seat 1).  Returns done,
  // or -1 (state untouched) for an illegal action.
  __device__ static int step(const DevEnv&, State& s, int a0, int a1, float& r0, float& r1,
                             float& team) {
    const int me = s.turn & 1, pa = me ^ 1;
    const int a = me == 0 ? a0 : a1;
    if (a < 0 || a >= 20 || !((legal(s) >> a) & 1u)) {
      r0 = r1 = team = 0.0f;
      return -1;
    }
    const int fr_start = s.fr;
    const int score_before = s.score;
    float reward = 0.0f;
    uint8_t flags = (uint8_t)(1u | (me << 1));
    s.la_colour = 255;
    s.la_rank = 0;
    s.la_slot = 255;
    s.la_card = 255;
    s.la_hinted = 0;
    if (a < 10) {
      const int slot = a % 5;
      const int card = s.hand[me][slot];
      const int c = card / 5, rank = card % 5 + 1;
      s.la_type = a < 5 ? 0 : 1;
      s.la_colour = (uint8_t)c;
      s.la_rank = (uint8_t)rank;
      s.la_slot = (uint8_t)slot;
      s.la_card = (uint8_t)card;
      remove_slot(s, me, slot);
      if (a < 5) {
        if (s.fw[c] == rank - 1) {
          s.fw[c] = (uint8_t)rank;
          s.score += 1;
          reward = 1.0f;
          if (rank == 5 && s.info < 8) s.info += 1;
          flags |= 4u;
        } else {
          s.lives -= 1;
          s.disc[card] += 1;
          flags |= 8u;
        }
      } else {
        s.disc[card] += 1;
        s.info += 1;
      }
      if (s.ptr < 50) {
        const int k = s.n_hand[me];
        s.hand[me][k] = s.deck[s.ptr];
        s.know[me][k] = 0x1FFFFFFu;
        s.hints[me][k] = 0;
        s.n_hand[me] = (uint8_t)(k + 1);
        s.ptr += 1;
        if (s.ptr == 50) s.fr = 2;
      }
    } else {
      const bool by_colour = a < 15;
      const int v = (a - 10) % 5;
      const uint32_t bits = by_colour ? colour_bits(v) : rank_bits(v);
      s.info -= 1;
      s.la_type = by_colour ? 2 : 3;
      if (by_colour) s.la_colour = (uint8_t)v;
      else s.la_rank = (uint8_t)(v + 1);
      uint8_t hinted = 0;
      for (int k = 0; k < s.n_hand[pa]; ++k) {
        const int card = s.hand[pa][k];
        if (by_colour ? (card / 5 == v) : (card % 5 == v)) {
          s.know[pa][k] &= bits;
          s.hints[pa][k] |= (uint16_t)(1u << (by_colour ? v : 5 + v));
          hinted |= (uint8_t)(1u << k);
        } else {
          s.know[pa][k] &= ~bits;
        }
      }
      s.la_hinted = hinted;
    }
    s.la_flags = flags;
    s.turn += 1;
    int done = 0;
    if (s.lives == 0) {
      done = 1;
      reward = -(float)score_before;
    } else if (s.score == 25) {
      done = 1;
    } else if (fr_start >= 1) {
      s.fr = (int8_t)(fr_start - 1);
      done = s.fr == 0;
    }
    if (!done && s.turn >= kTurnCap) done = 1;
    r0 = r1 = team = reward;
    s.ret = __fadd_rn(s.ret, reward);
    return done;
  }

  // 660 binary features for `seat` (see the section offsets below).
  template <class Row>
  __device__ static void obs_into(const DevEnv&, const State& s, int seat, Row& row) {
    row.clear();
    const int me = seat, pa = seat ^ 1;
    for (int k = 0; k < s.n_hand[pa]; ++k) row.set(k * 25 + s.hand[pa][k], 1);  // [0,125)
    for (int q = 0; q < 2; ++q) {                                              // [125,375)
      const int who = q == 0 ? me : pa;
      for (int k = 0; k < s.n_hand[who]; ++k) row.set_bits(125 + q * 125 + k * 25, s.know[who][k], 25);
    }
    for (int c = 0; c < 5; ++c)                                                // [375,400)
      if (s.fw[c]) row.set(375 + c * 5 + s.fw[c] - 1, 1);
    row.set_run(400, s.info);                                                  // [400,408)
    row.set_run(408, s.lives);                                                 // [408,411)
    row.set_run(411, 50 - s.ptr);                                              // [411,451)
    const uint8_t base[5] = {0, 3, 5, 7, 9};
    for (int t = 0; t < 25; ++t)                                               // [451,501)
      row.set_run(451 + (t / 5) * 10 + base[t % 5], s.disc[t]);
    if (s.la_flags & 1u) {                                                     // [501,554)
      const int o = 501;
      row.set(o + (((s.la_flags >> 1) & 1u) == (uint32_t)me ? 0 : 1), 1);
      row.set(o + 2 + s.la_type, 1);
      if (s.la_colour != 255) row.set(o + 6 + s.la_colour, 1);
      if (s.la_rank) row.set(o + 11 + s.la_rank - 1, 1);
      if (s.la_slot != 255) row.set(o + 16 + s.la_slot, 1);
      if (s.la_card != 255) row.set(o + 21 + s.la_card, 1);
      row.set_bits(o + 46, s.la_hinted, 5);
      if (s.la_flags & 4u) row.set(o + 51, 1);
      if (s.la_flags & 8u) row.set(o + 52, 1);
    }
    for (int q = 0; q < 2; ++q) {                                              // [554,654)
      const int who = q == 0 ? me : pa;
      for (int k = 0; k < 5; ++k) row.set_bits(554 + q * 50 + k * 10, s.hints[who][k], 10);
    }
    row.set_run(654, s.n_hand[me]);                                            // [654,659)
    if (s.fr >= 0) row.set(659, 1);                                            // [659]
  }
  // The same bits into a word row (the streamed cross-play kernel): every section is a
  // field of at most 64 bits at a fixed position, ORed into registers, one store per word.
  static constexpr int kObsWords = (660 + 31) / 32;
  __device__ static void obs_into(const DevEnv&, const State& s, int seat, ObsBits& row) {
    uint32_t wd[kObsWords];
#pragma unroll
    for (int i = 0; i < kObsWords; ++i) wd[i] = 0u;
    auto put = [&](int pos, int nbits, uint64_t v) {  // v < 2^nbits, nbits <= 64
      const int w = pos >> 5, sh = pos & 31;
      wd[w] |= (uint32_t)(v << sh);
      if (sh + nbits > 32) wd[w + 1] |= (uint32_t)((v << sh) >> 32);
      if (sh + nbits > 64) wd[w + 2] |= (uint32_t)(v >> (64 - sh));
    };
    const int me = seat, pa = seat ^ 1;
#pragma unroll
    for (int k = 0; k < 5; ++k)  // [0,125) the partner's cards, one-hot
      put(25 * k, 25, k < s.n_hand[pa] ? 1ull << s.hand[pa][k] : 0ull);
#pragma unroll
    for (int q = 0; q < 2; ++q) {  // [125,375) card knowledge, own then the partner's
      const int who = q == 0 ? me : pa;
#pragma unroll
      for (int k = 0; k < 5; ++k)
        put(125 + 125 * q + 25 * k, 25, k < s.n_hand[who] ? (uint64_t)(s.know[who][k] & 0x1FFFFFFu) : 0ull);
    }
    uint32_t fw = 0;  // [375,400) fireworks
#pragma unroll
    for (int c = 0; c < 5; ++c)
      if (s.fw[c]) fw |= 1u << (5 * c + s.fw[c] - 1);
    put(375, 25, fw);
    // [400,451) information tokens, life tokens, cards left in the deck (thermometers)
    put(400, 51, ((1ull << s.info) - 1) | (((1ull << s.lives) - 1) << 8) | (((1ull << (50 - s.ptr)) - 1) << 11));
    uint64_t disc = 0;  // [451,501) discards: a thermometer per card type (3, 2, 2, 2, 1 copies)
#pragma unroll
    for (int t = 0; t < 25; ++t) {
      const int base = (t % 5) == 0 ? 0 : (t % 5) == 1 ? 3 : (t % 5) == 2 ? 5 : (t % 5) == 3 ? 7 : 9;
      disc |= ((1ull << s.disc[t]) - 1) << ((t / 5) * 10 + base);
    }
    put(451, 50, disc);
    if (s.la_flags & 1u) {  // [501,554) the last action
      uint64_t la = 1ull << ((((s.la_flags >> 1) & 1u) == (uint32_t)me) ? 0 : 1);
      la |= 1ull << (2 + s.la_type);
      if (s.la_colour != 255) la |= 1ull << (6 + s.la_colour);
      if (s.la_rank) la |= 1ull << (11 + s.la_rank - 1);
      if (s.la_slot != 255) la |= 1ull << (16 + s.la_slot);
      if (s.la_card != 255) la |= 1ull << (21 + s.la_card);
      la |= (uint64_t)(s.la_hinted & 0x1Fu) << 46;
      if (s.la_flags & 4u) la |= 1ull << 51;
      if (s.la_flags & 8u) la |= 1ull << 52;
      put(501, 53, la);
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {  // [554,654) explicit hints, own then the partner's
      const int who = q == 0 ? me : pa;
#pragma unroll
      for (int k = 0; k < 5; ++k) put(554 + 50 * q + 10 * k, 10, s.hints[who][k] & 0x3FFu);
    }
    // [654,659) own hand size (thermometer), [659] the final round
    put(654, 6, ((1ull << s.n_hand[me]) - 1) | (s.fr >= 0 ? 1ull << 5 : 0ull));
#pragma unroll
    for (int i = 0; i < kObsWords; ++i) row.w[i] = wd[i];
    for (int i = kObsWords; i < row.words; ++i) row.w[i] = 0u;
  }
  __device__ static void obs(const DevEnv& d, const State& s, int seat, uint8_t* row) {
    ObsBytes w{row, 165};
    obs_into(d, s, seat, w);
  }

  __device__ static float ret(const State& s) { return s.ret; }
};

}  // namespace aht
