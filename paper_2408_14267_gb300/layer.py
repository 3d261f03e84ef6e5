"""One fully quantized layer step through the C-ABI (App. C, Algorithm 1).

`LayerStep` owns the device buffers of one linear or convolution layer and
enqueues, on one CUDA stream and without host synchronisation:

  forward : pack sign(W) (rows, columns, column sums); pack sign(X) or the
            Unfolder of X fused with sign; binarized GEMM, y = Gamma * acc.
            A stride-1 "same" convolution with C a multiple of 128 runs the
            implicit-GEMM forward instead: sign(X) packed per pixel, sign(W)
            packed tap-major, and the Unfolder writes only the column packing
            that grad_weight reads
  backward: SCQ quantization of G = gY (.) Gamma (ranges, AGP selection,
            stochastic rounding of both branches); grad_input GEMM (PSQ side)
            then, for a convolution, the Folder; grad_weight GEMM (PCQ side)

All arithmetic runs in libfqt1's kernels; this module only allocates and
passes pointers.  The weight update (Algorithm 1's last step) is not part of
the layer step.
"""
import numpy as np
import torch

from . import fqt1


def conv_out_hw(H, W, kh, kw, stride, pad):
    return (H + 2 * pad - kh) // stride + 1, (W + 2 * pad - kw) // stride + 1


class LayerStep:
    """Buffers and launches of one layer step.  keep_acc=False skips the optional
    int32 copy of the forward accumulators (the benchmark's configuration)."""

    def __init__(self, wl, device="cuda", keep_acc=True, fold=None, implicit=False, e4m3_weights=False,
                 e4m3_x=False, colmajor=None, acc16=True):
        dev = torch.device(device)
        self.kind = wl["kind"]
        self.keep_acc = keep_acc
        f32 = dict(dtype=torch.float32, device=dev)
        i32 = dict(dtype=torch.int32, device=dev)
        def dev_tensor(a):  # host arrays are copied in; device tensors are taken as they are
            if isinstance(a, torch.Tensor):
                return a.to(**f32).contiguous()
            return torch.as_tensor(np.ascontiguousarray(a), **f32)

        self.x = dev_tensor(wl["x"])
        self.w = dev_tensor(wl["w"])
        self.gamma = None if wl.get("gamma") is None else dev_tensor(wl["gamma"])
        self.gy = dev_tensor(wl["gy"])
        if self.kind == "conv":
            N, Cin, H, W = self.x.shape
            D, _, kh, kw = self.w.shape
            self.stride, self.pad = wl["stride"], wl["pad"]
            Ho, Wo = conv_out_hw(H, W, kh, kw, self.stride, self.pad)
            self.conv = (N, Cin, H, W, kh, kw)
            M, K, rpg = N * Ho * Wo, Cin * kh * kw, Ho * Wo
        else:
            M, K = self.x.shape
            D = self.w.shape[0]
            rpg = wl.get("rows_per_group", 1)
        self.M, self.K, self.D, self.rpg = M, K, D, rpg
        # convolutions whose samples fit a 128-row tile fold grad_input in the GEMM epilogue,
        # unless the int32 accumulators are kept (keep_acc) or fold is forced off
        if self.kind == "conv":
            ok = fqt1.fold_supported(Ho, Wo, kh, kw, H, W)
            self.fold = (not keep_acc and ok) if fold is None else (fold and ok)
        else:
            self.fold = False
        # convolutions without the fused Folder: grad_input through column-major int32
        # accumulators and the column-major Folder (every tap read as contiguous runs), unless
        # the row-major accumulators are kept (keep_acc) or colmajor is forced off
        if self.kind == "conv" and not self.fold:
            self.colmajor = (not keep_acc) if colmajor is None else bool(colmajor)
        else:
            self.colmajor = False
        # implicit-GEMM forward on request, where the library supports the convolution (off by
        # default: on the 8 x 8, 256-channel layer its two extra packing kernels cost more than
        # the Unfolder's row packing they replace)
        if self.kind == "conv":
            self.implicit = bool(implicit) and fqt1.conv_implicit_supported(N, Cin, H, W, kh, kw, self.stride,
                                                                              self.pad)
        else:
            self.implicit = False
        wK, wM, wD = fqt1.packed_words(K), fqt1.packed_words(M), fqt1.packed_words(D)
        # shapes whose Unfolder reads an input region per tile: sign-pack x into planes first
        # (one streaming pass), so that the regions are read as bits
        self.x_planes = None
        if self.kind == "conv" and not self.implicit and fqt1.unfold_from_planes(N, Cin, H, W, kh, kw, self.stride,
                                                                                 self.pad):
            self.x_planes = torch.empty(N * Cin * fqt1.plane_words(H, W), **i32)
        if self.implicit:
            self.x_pix = torch.empty(N * H * W, fqt1.packed_words(Cin), **i32)
            self.w_taps = torch.empty(D, wK, **i32)
        # e4m3 copies of sign(X_u) (rows for the forward product, columns for grad_weight's),
        # written by the Unfolder instead of the packed words: both products then load their
        # sign operand by TMA and expand nothing.  Where the whole-image Unfolder serves the
        # convolution (fqt1_im2col_path 2), or for a linear layer whose rows are a multiple of 4
        # floats; the forward then takes the e4m3 copy of sign(W) too
        u8 = dict(dtype=torch.uint8, device=dev)
        self.e4m3_x = False
        if e4m3_x and not self.implicit:
            if self.kind == "conv":
                self.e4m3_x = fqt1.im2col_path(N, Cin, H, W, kh, kw, self.stride, self.pad) == 2
            else:
                self.e4m3_x = K % 4 == 0
        if self.e4m3_x:
            self.x_planes = None
            self.x8_row = torch.empty(M, fqt1.codes_ld(K), **u8)
            self.x8_col = torch.empty(K, fqt1.codes_ld(M), **u8)
            e4m3_weights = True if e4m3_weights is True or e4m3_weights == "fold" else "fwd"
        self.sx_row = None if self.implicit or self.e4m3_x else torch.empty(M, wK, **i32)
        self.sx_col = None if self.e4m3_x else torch.empty(K, wM, **i32)
        self.cs_x = torch.empty(K, **i32)
        self.sw_row = None if self.implicit else torch.empty(D, wK, **i32)
        # e4m3 copies of sign(W) (rows for the forward product, columns for the fused Folder's
        # product): B then goes to the tensor cores by TMA instead of being expanded per CTA.
        # Off by default: on the 8 x 8, 256-channel layer the step graph is as fast either way
        # e4m3_weights: True (both products), "fwd" or "fold" (one of them), False
        e_fwd = e4m3_weights is True or e4m3_weights == "fwd"
        e_fold = e4m3_weights is True or e4m3_weights == "fold"
        self.w8 = torch.empty(D, fqt1.codes_ld(K), **u8) if e_fwd and not self.implicit else None
        self.wt8 = torch.empty(K, fqt1.codes_ld(D), **u8) if e_fold and self.fold else None
        # e4m3 sign(W)^T for the column-major product on request only (e4m3_weights="colmajor"):
        # measured no faster than the packed signs there
        if e4m3_weights == "colmajor" and self.colmajor:
            self.wt8 = torch.empty(K, fqt1.codes_ld(D), **u8)
        self.sw_col = torch.empty(K, wD, **i32)
        self.cs_w = torch.empty(K, **i32)
        self.acc_y = torch.empty(M, D, **i32) if keep_acc else None
        # without a Gamma the forward uses unit scales and G = gY
        self.gamma_fwd = self.gamma if self.gamma is not None else torch.ones(D, **f32)
        self.y = torch.empty(M, D, **f32)
        self.p_s = fqt1.AgpParams(wl["bits_s"], wl["mode_s"], wl["seed_s"], rpg)
        self.p_c = fqt1.AgpParams(wl["bits_c"], wl["mode_c"], wl["seed_c"], 1)
        n_s = M // rpg
        self.cap_s = fqt1.kept_capacity(n_s, wl["bits_s"], wl["mode_s"])
        self.cap_c = fqt1.kept_capacity(D, wl["bits_c"], wl["mode_c"])
        self.psq = fqt1.QGradBuffers(n_s, self.cap_s, self.cap_s * rpg, D, dev)
        self.pcq = fqt1.QGradBuffers(D, self.cap_c, self.cap_c, M, dev)
        self.ws = fqt1.scq_workspace(M, D, K, rpg, dev)
        self.dev_status = torch.zeros(4, **i32)
        self.acc_dx = torch.empty(max(self.cap_s * rpg, 1), K, **i32)
        # column-major accumulators for the column-major Folder: [K][ld_cm], ld_cm >= kept rows, a
        # multiple of 32 so that every column starts on a 128-byte line; int16 where every sum
        # fits (acc_bits_cm: (2^b - 1) D <= 32767), which halves their traffic, else int32
        self.ld_cm = (max(self.cap_s * rpg, 1) + 31) // 32 * 32
        self.acc_bits_cm = fqt1.colmajor_acc_bits(wl["bits_s"], D) if acc16 else 32
        cm_type = torch.int16 if self.acc_bits_cm == 16 else torch.int32
        self.acc_dx_cm = torch.empty(K, self.ld_cm, dtype=cm_type, device=dev) if self.colmajor else None
        self.dx = torch.empty(*(self.x.shape), **f32)
        self.acc_dw = torch.empty(max(self.cap_c, 1), K, **i32)
        self.dw = torch.empty(D, K, **f32)

    # dense-equivalent operations of one step: forward, grad_input and grad_weight products
    def dense_ops(self):
        return 6.0 * self.M * self.K * self.D

    FORWARD_STAGES = ("pack_w", "pack_xp", "pack_x", "im2col", "fwd_gemm")

    def stages(self):
        """The step as (name, launch(stream)) pairs, in stream order."""
        if self.implicit:
            N, Cin, H, W, kh, kw = self.conv

            def pack_w(s):
                if self.wt8 is not None:
                    fqt1.binarize_pack_e4m3(self.w, self.D, self.K, self.K, None, self.sw_col, self.cs_w, None,
                                            self.wt8, s)
                else:
                    fqt1.binarize_pack(self.w, self.D, self.K, self.K, None, self.sw_col, self.cs_w, s)
                fqt1.pack_weight_taps(self.w, self.D, Cin, kh, kw, self.w_taps, s)

            st = [("pack_w", pack_w),
                  ("pack_xp", lambda s: fqt1.pack_pixels(self.x, N, Cin, H, W, self.x_pix, s)),
                  ("im2col", lambda s: fqt1.im2col(self.x, N, Cin, H, W, kh, kw, self.stride, self.pad, None,
                                                   self.sx_col, self.cs_x, s)),
                  ("fwd_gemm", lambda s: fqt1.conv_fwd_implicit(self.x_pix, self.w_taps, N, Cin, H, W, kh, kw,
                                                                self.stride, self.pad, self.D, self.gamma_fwd, None,
                                                                self.acc_y, self.y, s))]
        else:
            def pack_w(s):
                if self.w8 is not None or self.wt8 is not None:  # the e4m3 copies from the same pass
                    fqt1.binarize_pack_e4m3(self.w, self.D, self.K, self.K, self.sw_row, self.sw_col, self.cs_w,
                                            self.w8, self.wt8, s)
                else:
                    fqt1.binarize_pack(self.w, self.D, self.K, self.K, self.sw_row, self.sw_col, self.cs_w, s)

            st = [("pack_w", pack_w)]
            if self.e4m3_x and self.kind == "conv":
                N, Cin, H, W, kh, kw = self.conv
                st.append(("im2col", lambda s: fqt1.im2col_e4m3(self.x, N, Cin, H, W, kh, kw, self.stride, self.pad,
                                                                self.x8_row, self.x8_col, self.cs_x, s)))
            elif self.e4m3_x:
                st.append(("pack_x", lambda s: fqt1.binarize_pack_e4m3(self.x, self.M, self.K, self.K, None, None,
                                                                       self.cs_x, self.x8_row, self.x8_col, s)))
            elif self.kind == "conv" and self.x_planes is not None:
                N, Cin, H, W, kh, kw = self.conv

                def unfold(s):
                    fqt1.pack_planes(self.x, N, Cin, H, W, self.x_planes, s)
                    fqt1.im2col_planes(self.x_planes, N, Cin, H, W, kh, kw, self.stride, self.pad, self.sx_row,
                                       self.sx_col, self.cs_x, s)
                st.append(("im2col", unfold))
            elif self.kind == "conv":
                N, Cin, H, W, kh, kw = self.conv
                st.append(("im2col", lambda s: fqt1.im2col(self.x, N, Cin, H, W, kh, kw, self.stride, self.pad,
                                                           self.sx_row, self.sx_col, self.cs_x, s)))
            else:
                st.append(("pack_x", lambda s: fqt1.binarize_pack(self.x, self.M, self.K, self.K, self.sx_row,
                                                                  self.sx_col, self.cs_x, s)))
            if self.e4m3_x:
                st.append(("fwd_gemm", lambda s: fqt1.fwd_gemm_e4m3x(self.x8_row, self.w8, self.M, self.D, self.K,
                                                                     self.gamma_fwd, None, self.acc_y, self.y, s)))
            elif self.w8 is not None:
                st.append(("fwd_gemm", lambda s: fqt1.fwd_gemm_e4m3w(self.sx_row, self.w8, self.M, self.D, self.K,
                                                                     self.gamma_fwd, None, self.acc_y, self.y, s)))
            else:
                st.append(("fwd_gemm", lambda s: fqt1.fwd_gemm(self.sx_row, self.sw_row, self.M, self.D, self.K,
                                                               self.gamma_fwd, self.acc_y, self.y, s)))
        st.append(("scq_quantize", lambda s: fqt1.scq_quantize(self.gy, self.M, self.D, self.gamma, self.p_s,
                                                               self.p_c, self.psq, self.pcq, self.ws,
                                                               self.dev_status, s)))
        if self.kind == "conv" and self.fold:
            N, Cin, H, W, kh, kw = self.conv
            if self.wt8 is not None:
                st.append(("bwd_input_fold", lambda s: fqt1.bwd_input_fold_e4m3w(self.psq, self.wt8, self.cs_w, N, Cin,
                                                                                 H, W, kh, kw, self.stride, self.pad,
                                                                                 self.D, self.p_s, self.dx, s)))
            else:
                st.append(("bwd_input_fold", lambda s: fqt1.bwd_input_fold(self.psq, self.sw_col, self.cs_w, N, Cin,
                                                                           H, W, kh, kw, self.stride, self.pad,
                                                                           self.D, self.p_s, self.dx, s)))
        elif self.kind == "conv" and self.colmajor:
            N, Cin, H, W, kh, kw = self.conv
            if self.wt8 is not None:
                st.append(("bwd_input_gemm", lambda s: fqt1.bwd_input_gemm_colmajor_e4m3w(
                    self.psq, self.wt8, self.M, self.D, self.K, self.p_s, self.acc_dx_cm, s)))
            else:
                st.append(("bwd_input_gemm", lambda s: fqt1.bwd_input_gemm_colmajor(
                    self.psq, self.sw_col, self.M, self.D, self.K, self.p_s, self.acc_dx_cm, s)))
            st.append(("col2im", lambda s: fqt1.col2im_colmajor(self.acc_dx_cm, self.psq, self.cs_w, N, Cin, H, W, kh,
                                                                kw, self.stride, self.pad, self.dx, s)))
        elif self.kind == "conv":
            N, Cin, H, W, kh, kw = self.conv
            st.append(("bwd_input_gemm", lambda s: fqt1.bwd_input_gemm(self.psq, self.sw_col, self.cs_w, self.M,
                                                                       self.D, self.K, self.p_s, self.acc_dx, None,
                                                                       s)))
            st.append(("col2im", lambda s: fqt1.col2im(self.acc_dx, self.psq, self.cs_w, N, Cin, H, W, kh, kw,
                                                       self.stride, self.pad, self.dx, s)))
        else:
            # without keep_acc the dequantization runs in the GEMM epilogue (no int32 round trip)
            acc = self.acc_dx if self.keep_acc else None
            st.append(("bwd_input_gemm", lambda s: fqt1.bwd_input_gemm(self.psq, self.sw_col, self.cs_w, self.M,
                                                                       self.D, self.K, self.p_s, acc, self.dx, s)))
        if self.e4m3_x:
            st.append(("bwd_weight_gemm", lambda s: fqt1.bwd_weight_gemm_e4m3x(self.pcq, self.x8_col, self.cs_x,
                                                                               self.M, self.D, self.K, self.p_c,
                                                                               self.acc_dw, self.dw, s)))
        else:
            st.append(("bwd_weight_gemm", lambda s: fqt1.bwd_weight_gemm(self.pcq, self.sx_col, self.cs_x, self.M,
                                                                         self.D, self.K, self.p_c, self.acc_dw,
                                                                         self.dw, None, s)))
        return st

    def forward(self, stream=None):
        for name, fn in self.stages():
            if name in self.FORWARD_STAGES:
                fn(stream)

    def backward(self, stream=None):
        for name, fn in self.stages():
            if name not in self.FORWARD_STAGES:
                fn(stream)

    def step(self, stream=None):
        for name, fn in self.stages():
            fn(stream)

    def step_concurrent(self, stream=None):
        """The same step as three stream branches joined by events (capturable in one graph).

        The packing of W, the packing / Unfolder of X and the SCQ quantization of gY are
        independent; each product waits only for its own operands:
          calling stream: pack X -> (wait W) forward -> (wait SCQ) grad_weight -> join
          branch 1      : pack W
          branch 2      : SCQ quantize -> (wait W) grad_input (-> Folder)
        With the implicit-GEMM forward the calling stream packs X per pixel, and the Unfolder
        (only grad_weight reads its column packing) runs on branch 1 after pack W.
        """
        main = stream if stream is not None else torch.cuda.current_stream()
        if not hasattr(self, "_branches"):
            self._branches = (torch.cuda.Stream(device=main.device), torch.cuda.Stream(device=main.device))
        b1, b2 = self._branches
        st = dict(self.stages())
        fork = torch.cuda.Event()
        fork.record(main)
        b1.wait_event(fork)
        b2.wait_event(fork)
        st["pack_w"](b1)
        w_ready = torch.cuda.Event()
        w_ready.record(b1)
        st["scq_quantize"](b2)
        q_ready = torch.cuda.Event()
        q_ready.record(b2)
        b2.wait_event(w_ready)
        if "bwd_input_fold" in st:
            st["bwd_input_fold"](b2)
        else:
            st["bwd_input_gemm"](b2)
            if "col2im" in st:
                st["col2im"](b2)
        if self.implicit:
            st["im2col"](b1)
            x_ready = torch.cuda.Event()
            x_ready.record(b1)
            st["pack_xp"](main)
        else:
            st["im2col" if "im2col" in st else "pack_x"](main)
        main.wait_event(w_ready)
        st["fwd_gemm"](main)
        main.wait_event(q_ready)
        if self.implicit:
            main.wait_event(x_ready)
        st["bwd_weight_gemm"](main)
        b2_done = torch.cuda.Event()
        b2_done.record(b2)
        main.wait_event(b2_done)

    def step_concurrent_host(self, h_in, h_out, stream=None):
        """step_concurrent with the host copies of one step, capturable in one graph.

        h_in: pinned host tensors (x, w, gy[, gamma]) copied into the layer's inputs; h_out:
        pinned host tensors (y, dx, dw) that receive the outputs.  The host link carries one
        copy at a time at full rate (parallel copies share it), so the copies run in a fixed
        order on two streams and each branch starts as soon as its own input has landed:
          copies in : W, Gamma (if any), gY, X
          branch 1  : (W in) pack W
          branch 2  : (gY in) SCQ quantize -> (W packed) grad_input (-> Folder)
          calling   : (X in) pack / Unfolder -> (W packed) forward -> (SCQ) grad_weight
          (implicit-GEMM forward: the calling stream packs X per pixel and branch 1 runs the
          Unfolder after pack W and X in; grad_weight also waits for it)
          copies out: (all in, grad_input done) dx, (forward done) y, (grad_weight done) dw
        """
        main = stream if stream is not None else torch.cuda.current_stream()
        if not hasattr(self, "_branches4"):
            self._branches4 = tuple(torch.cuda.Stream(device=main.device) for _ in range(4))
        b1, b2, cin, cout = self._branches4
        st = dict(self.stages())

        def ev(s):
            e = torch.cuda.Event()
            e.record(s)
            return e

        fork = ev(main)
        for b in (b1, b2, cin, cout):
            b.wait_event(fork)
        x_h, w_h, gy_h = h_in[0], h_in[1], h_in[2]
        g_h = h_in[3] if len(h_in) > 3 else None
        with torch.cuda.stream(cin):
            self.w.copy_(w_h, non_blocking=True)
            w_in = ev(cin)
            if g_h is not None:
                self.gamma.copy_(g_h, non_blocking=True)
            self.gy.copy_(gy_h, non_blocking=True)
            gy_in = ev(cin)
            self.x.copy_(x_h, non_blocking=True)
            x_in = ev(cin)
        b1.wait_event(w_in)
        st["pack_w"](b1)
        w_ready = ev(b1)
        b2.wait_event(gy_in)
        st["scq_quantize"](b2)
        q_ready = ev(b2)
        b2.wait_event(w_ready)
        if "bwd_input_fold" in st:
            st["bwd_input_fold"](b2)
        else:
            st["bwd_input_gemm"](b2)
            if "col2im" in st:
                st["col2im"](b2)
        dx_ready = ev(b2)
        main.wait_event(x_in)
        if self.implicit:  # the Unfolder feeds only grad_weight: branch 1, after pack W
            b1.wait_event(x_in)
            st["im2col"](b1)
            x_ready = ev(b1)
            st["pack_xp"](main)
        else:
            st["im2col" if "im2col" in st else "pack_x"](main)
        main.wait_event(w_ready)
        main.wait_event(gy_in)  # Gamma (copied before gY) scales the forward
        st["fwd_gemm"](main)
        y_ready = ev(main)
        main.wait_event(q_ready)
        if self.implicit:
            main.wait_event(x_ready)
        st["bwd_weight_gemm"](main)
        dw_ready = ev(main)
        cout.wait_event(x_in)  # the outputs follow the inputs on the link
        with torch.cuda.stream(cout):
            cout.wait_event(dx_ready)
            h_out[1].copy_(self.dx, non_blocking=True)
            cout.wait_event(y_ready)
            h_out[0].copy_(self.y, non_blocking=True)
            cout.wait_event(dw_ready)
            h_out[2].copy_(self.dw, non_blocking=True)
        main.wait_event(ev(cout))
        main.wait_event(ev(b2))
