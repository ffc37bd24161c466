// env_minihanabi.cuh -- 2-player Mini Hanabi on the device (one thread per env).
//
// 3 colours x ranks 1,1,1,2,2,3 (18 cards), 2-card hands, 3 info and 1 life tokens, 10
// actions (play slot 0-1, discard slot 0-1, hint colour 0-2, hint rank 1-3), seat 0
// first.  Card type = colour*3 + rank-1.  The full game's rules at this size (Sec. 4
// Table: "Mini (3 colors x 3 ranks)"); the observation is the full game's sections at
// this size, 153 features, then 3 zero features (156).
#pragma once
#include "aht_common.cuh"

namespace aht {

struct EnvMiniHanabi {
  static constexpr bool kTurnBased = true;
  static constexpr int kNumActions = 10;
  static constexpr int kTurnCap = 100;
  struct State {
    uint8_t deck[20];       // 18 used
    uint8_t hand[2][2];
    uint8_t n_hand[2];
    uint16_t know[2][2];    // possible card types, 9 bits
    uint8_t hints[2][2];    // explicit hints received: bits 0-2 colour, 3-5 rank
    uint8_t fw[3], info, lives, score, ptr, turn;
    uint8_t disc[9];
    int8_t fr;              // final-round turns left, -1 while the deck has cards
    uint8_t la_flags;       // bit0 valid, bit1 actor seat, bit2 play success, bit3 bomb
    uint8_t la_type, la_colour, la_rank, la_slot, la_card, la_hinted;
    uint8_t pad[2];
    float ret;
  };
  static constexpr int kWords = sizeof(State) / 4;
  static_assert(sizeof(State) % 4 == 0, "state words");

  __device__ static uint32_t colour_bits(int c) { return 0x7u << (3 * c); }
  __device__ static uint32_t rank_bits(int r0) { return 0x49u << r0; }  // rank index 0..2

  __device__ static void reset(const DevEnv&, Key key, uint32_t env, uint32_t step, State& s) {
    for (int c = 0; c < 3; ++c) {  // canonical order: colour c, ranks 1,1,1,2,2,3
      uint8_t* p = s.deck + c * 6;
      const uint8_t b = (uint8_t)(c * 3);
      p[0] = p[1] = p[2] = b;
      p[3] = p[4] = b + 1;
      p[5] = b + 2;
    }
    s.deck[18] = s.deck[19] = 0;
    DrawSeq r(key, env, step, kStreamReset);
    for (int i = 17; i >= 1; --i) {
      const int j = (int)uniform_int(r.next(), (uint32_t)(i + 1));
      const uint8_t t = s.deck[i];
      s.deck[i] = s.deck[j];
      s.deck[j] = t;
    }
    for (int p = 0; p < 2; ++p) {
      for (int k = 0; k < 2; ++k) {
        s.hand[p][k] = s.deck[p * 2 + k];
        s.know[p][k] = 0x1FFu;
        s.hints[p][k] = 0;
      }
      s.n_hand[p] = 2;
    }
    for (int c = 0; c < 3; ++c) s.fw[c] = 0;
    for (int t = 0; t < 9; ++t) s.disc[t] = 0;
    s.info = 3;
    s.lives = 1;
    s.score = 0;
    s.ptr = 4;
    s.turn = 0;
    s.fr = -1;
    s.la_flags = 0;
    s.la_type = s.la_colour = s.la_rank = s.la_slot = s.la_card = s.la_hinted = 0;
    s.pad[0] = s.pad[1] = 0;
    s.ret = 0.0f;
  }

  __device__ static int actor(const State& s) { return s.turn & 1; }

  __device__ static uint32_t legal(const State& s) {
    const int me = s.turn & 1, pa = me ^ 1;
    uint32_t m = 0;
    for (int k = 0; k < s.n_hand[me]; ++k) {
      m |= 1u << k;
      if (s.info < 3) m |= 1u << (2 + k);
    }
    if (s.info > 0) {
      for (int k = 0; k < s.n_hand[pa]; ++k) {
        const int card = s.hand[pa][k];
        m |= 1u << (4 + card / 3);
        m |= 1u << (7 + card % 3);
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
    if (a < 0 || a >= kNumActions || !((legal(s) >> a) & 1u)) {
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
    if (a < 4) {
      const int slot = a & 1;
      const int card = s.hand[me][slot];
      const int c = card / 3, rank = card % 3 + 1;
      s.la_type = a < 2 ? 0 : 1;
      s.la_colour = (uint8_t)c;
      s.la_rank = (uint8_t)rank;
      s.la_slot = (uint8_t)slot;
      s.la_card = (uint8_t)card;
      remove_slot(s, me, slot);
      if (a < 2) {
        if (s.fw[c] == rank - 1) {
          s.fw[c] = (uint8_t)rank;
          s.score += 1;
          reward = 1.0f;
          if (rank == 3 && s.info < 3) s.info += 1;
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
      if (s.ptr < 18) {
        const int k = s.n_hand[me];
        s.hand[me][k] = s.deck[s.ptr];
        s.know[me][k] = 0x1FFu;
        s.hints[me][k] = 0;
        s.n_hand[me] = (uint8_t)(k + 1);
        s.ptr += 1;
        if (s.ptr == 18) s.fr = 2;
      }
    } else {
      const bool by_colour = a < 7;
      const int v = (a - 4) % 3;
      const uint32_t bits = by_colour ? colour_bits(v) : rank_bits(v);
      s.info -= 1;
      s.la_type = by_colour ? 2 : 3;
      if (by_colour) s.la_colour = (uint8_t)v;
      else s.la_rank = (uint8_t)(v + 1);
      uint8_t hinted = 0;
      for (int k = 0; k < s.n_hand[pa]; ++k) {
        const int card = s.hand[pa][k];
        if (by_colour ? (card / 3 == v) : (card % 3 == v)) {
          s.know[pa][k] = (uint16_t)(s.know[pa][k] & bits);
          s.hints[pa][k] |= (uint8_t)(1u << (by_colour ? v : 3 + v));
          hinted |= (uint8_t)(1u << k);
        } else {
          s.know[pa][k] = (uint16_t)(s.know[pa][k] & ~bits);
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
    } else if (s.score == 9) {
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

  // 156 binary features for `seat` (153 + 3 zero; section offsets below).
  template <class Row>
  __device__ static void obs_into(const DevEnv&, const State& s, int seat, Row& row) {
    row.clear();
    const int me = seat, pa = seat ^ 1;
    for (int k = 0; k < s.n_hand[pa]; ++k) row.set(k * 9 + s.hand[pa][k], 1);   // [0,18)
    for (int q = 0; q < 2; ++q) {                                            // [18,54)
      const int who = q == 0 ? me : pa;
      for (int k = 0; k < s.n_hand[who]; ++k) row.set_bits(18 + q * 18 + k * 9, s.know[who][k], 9);
    }
    for (int c = 0; c < 3; ++c)                                              // [54,63)
      if (s.fw[c]) row.set(54 + c * 3 + s.fw[c] - 1, 1);
    row.set_run(63, s.info);                                                 // [63,66)
    row.set_run(66, s.lives);                                                // [66]
    row.set_run(67, 18 - s.ptr);                                             // [67,81)
    for (int t = 0; t < 9; ++t)                                              // [81,99)
      row.set_run(81 + (t / 3) * 6 + ((t % 3) == 0 ? 0 : ((t % 3) == 1 ? 3 : 5)), s.disc[t]);
    if (s.la_flags & 1u) {                                                   // [99,126)
      const int o = 99;
      row.set(o + (((s.la_flags >> 1) & 1u) == (uint32_t)me ? 0 : 1), 1);
      row.set(o + 2 + s.la_type, 1);
      if (s.la_colour != 255) row.set(o + 6 + s.la_colour, 1);
      if (s.la_rank) row.set(o + 9 + s.la_rank - 1, 1);
      if (s.la_slot != 255) row.set(o + 12 + s.la_slot, 1);
      if (s.la_card != 255) row.set(o + 14 + s.la_card, 1);
      row.set_bits(o + 23, s.la_hinted, 2);
      if (s.la_flags & 4u) row.set(o + 25, 1);
      if (s.la_flags & 8u) row.set(o + 26, 1);
    }
    for (int q = 0; q < 2; ++q) {                                            // [126,150)
      const int who = q == 0 ? me : pa;
      for (int k = 0; k < 2; ++k) row.set_bits(126 + q * 12 + k * 6, s.hints[who][k], 6);
    }
    row.set_run(150, s.n_hand[me]);                                          // [150,152)
    if (s.fr >= 0) row.set(152, 1);                                          // [152]
  }
  // The same bits into a word row (the streamed cross-play kernel): each section a field
  // at its fixed position, ORed into register words, one store per word.
  static constexpr int kObsWords = (156 + 31) / 32;
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
    for (int k = 0; k < 2; ++k)  // [0,18) the partner's cards, one-hot
      put(9 * k, 9, k < s.n_hand[pa] ? 1ull << s.hand[pa][k] : 0ull);
#pragma unroll
    for (int q = 0; q < 2; ++q) {  // [18,54) card knowledge, own then the partner's
      const int who = q == 0 ? me : pa;
#pragma unroll
      for (int k = 0; k < 2; ++k) put(18 + 18 * q + 9 * k, 9, k < s.n_hand[who] ? (uint64_t)(s.know[who][k] & 0x1FFu) : 0ull);
    }
    uint32_t fw = 0;  // [54,63) fireworks
#pragma unroll
    for (int c = 0; c < 3; ++c)
      if (s.fw[c]) fw |= 1u << (3 * c + s.fw[c] - 1);
    put(54, 9, fw);
    // [63,81) information tokens, life token, cards left in the deck (thermometers)
    put(63, 18, ((1ull << s.info) - 1) | (((1ull << s.lives) - 1) << 3) | (((1ull << (18 - s.ptr)) - 1) << 4));
    uint64_t disc = 0;  // [81,99) discards: a thermometer per card type (3, 2, 1 copies)
#pragma unroll
    for (int t = 0; t < 9; ++t)
      disc |= ((1ull << s.disc[t]) - 1) << ((t / 3) * 6 + ((t % 3) == 0 ? 0 : ((t % 3) == 1 ? 3 : 5)));
    put(81, 18, disc);
    if (s.la_flags & 1u) {  // [99,126) the last action
      uint64_t la = 1ull << ((((s.la_flags >> 1) & 1u) == (uint32_t)me) ? 0 : 1);
      la |= 1ull << (2 + s.la_type);
      if (s.la_colour != 255) la |= 1ull << (6 + s.la_colour);
      if (s.la_rank) la |= 1ull << (9 + s.la_rank - 1);
      if (s.la_slot != 255) la |= 1ull << (12 + s.la_slot);
      if (s.la_card != 255) la |= 1ull << (14 + s.la_card);
      la |= (uint64_t)(s.la_hinted & 0x3u) << 23;
      if (s.la_flags & 4u) la |= 1ull << 25;
      if (s.la_flags & 8u) la |= 1ull << 26;
      put(99, 27, la);
    }
#pragma unroll
    for (int q = 0; q < 2; ++q) {  // [126,150) explicit hints, own then the partner's
      const int who = q == 0 ? me : pa;
#pragma unroll
      for (int k = 0; k < 2; ++k) put(126 + 12 * q + 6 * k, 6, s.hints[who][k] & 0x3Fu);
    }
    // [150,152) own hand size (thermometer), [152] the final round
    put(150, 3, ((1ull << s.n_hand[me]) - 1) | (s.fr >= 0 ? 1ull << 2 : 0ull));
#pragma unroll
    for (int i = 0; i < kObsWords; ++i) row.w[i] = wd[i];
    for (int i = kObsWords; i < row.words; ++i) row.w[i] = 0u;
  }
  __device__ static void obs(const DevEnv& d, const State& s, int seat, uint8_t* row) {
    ObsBytes w{row, 39};
    obs_into(d, s, seat, w);
  }

  __device__ static float ret(const State& s) { return s.ret; }
};

}  // namespace aht
